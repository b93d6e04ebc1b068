"""Backward of the descriptor (dE/dT from dE/dD) on the GPU vs the oracle, and the full chain
dE/dD -> dE/dT -> (dE/ds, dE/dR~) against the oracle's chain (GPU)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import NP, TOL, lib, need_gpu, oracle_tables, product_model, rel, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _r32(a, dtype):
    return a.astype(np.float32).astype(np.float64) if dtype == torch.float32 else a


@pytest.mark.parametrize("nloc,M1,M2", [(37, 100, 16), (5, 37, 5), (3, 8, 8), (1, 1, 1), (130, 32, 4), (9, 256, 32)])
@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_descriptor_grad(nloc, M1, M2, dtype):
    dpc = lib()
    T = W.normal(1000 + M1, (nloc, 4, M1))
    dD = W.normal(2000 + M2, (nloc, M1, M2))
    Tg = torch.from_numpy(T.astype(NP[dtype])).cuda()
    dDg = torch.from_numpy(dD.astype(NP[dtype])).cuda()
    dT = dpc.dp_descriptor_contract_grad(Tg, dDg)
    torch.cuda.synchronize()
    ref = oracle.default().descriptor_grad(_r32(T, dtype), _r32(dD, dtype))
    assert rel(dT.double().cpu().numpy(), ref) <= TOL[dtype]


def test_descriptor_grad_empty():
    dpc = lib()
    T = torch.empty((0, 4, 16), dtype=torch.float64, device="cuda")
    dD = torch.empty((0, 16, 4), dtype=torch.float64, device="cuda")
    assert dpc.dp_descriptor_contract_grad(T, dD).shape == (0, 4, 16)


@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_full_chain_from_dD(dtype):
    """E's gradient from dE/dD all the way to dE/ds and dE/dR~: descriptor backward then fusion backward."""
    dpc = lib()
    w = W.water(seed=44, nmol=200)
    model = product_model(w, dtype)
    x = to_dev(w, dtype)
    dD = W.normal(77, (w.nloc, w.M1, w.M2))
    T = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    dT = dpc.dp_descriptor_contract_grad(T, torch.from_numpy(dD.astype(NP[dtype])).cuda())
    ds, dRt = dpc.dp_tabulate_fusion_grad(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel, dT)
    torch.cuda.synchronize()
    o = oracle.default()
    info, tabs = oracle_tables(w, dtype)
    s, Rt = _r32(w.s, dtype), _r32(w.Rt, dtype)
    Tr = o.fwd(tabs, info, s, Rt, w.nvalid, w.atype, w.sel)
    dTr = o.descriptor_grad(Tr, _r32(dD, dtype))
    dsr, dRr = o.grad(tabs, info, s, Rt, w.nvalid, w.atype, w.sel, dTr)
    tol = TOL[dtype] * (1 if dtype == torch.float64 else 5)
    assert rel(dT.double().cpu().numpy(), dTr) <= tol
    assert rel(ds.double().cpu().numpy(), dsr) <= tol
    assert rel(dRt.double().cpu().numpy(), dRr) <= tol


@pytest.mark.parametrize("widths,M2", [((1, 25, 50, 100), 16), ((1, 5, 37), 5), ((1, 8, 16, 32), 32), ((1, 7), 7),
                                       ((1, 7), 3), ((1, 64, 128, 256), 32), ((1, 16, 32, 64), 1)])
@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_fused_forward_descriptor(widths, M2, dtype):
    """T and D from one pass equal the oracle's T and D."""
    dpc = lib()
    w = W.tiny(seed=5 + M2, nloc=19, nreal=23, sel=31, widths=widths, M2=M2)
    model = product_model(w, dtype)
    x = to_dev(w, dtype)
    T, D = dpc.dp_tabulate_fusion_fwd_descriptor(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"],
                                                  w.sel, M2)
    torch.cuda.synchronize()
    o = oracle.default()
    info, tabs = oracle_tables(w, dtype)
    Tr = o.fwd(tabs, info, _r32(w.s, dtype), _r32(w.Rt, dtype), w.nvalid, w.atype, w.sel)
    assert rel(T.double().cpu().numpy(), Tr) <= TOL[dtype]
    assert rel(D.double().cpu().numpy(), o.descriptor(Tr, M2)) <= TOL[dtype]


def test_fused_forward_descriptor_limits():
    dpc = lib()
    w = W.tiny(seed=3, nloc=4, nreal=5, sel=8, widths=(1, 64), M2=33)
    model = product_model(w, torch.float64)
    x = to_dev(w, torch.float64)
    with pytest.raises(dpc.DPError) as e:
        dpc.dp_tabulate_fusion_fwd_descriptor(model.table, model.info, x["s"], x["Rt"], x["nvalid"], None, w.sel, 33)
    assert e.value.code == dpc.DP_ERR_UNSUPPORTED
