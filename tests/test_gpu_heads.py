"""Vector and tensor heads (the compressed path carried over to DP models of vectors and tensors, as
the paper's conclusion states) and the fitting net with several outputs on the GPU against the
oracle; the whole vector and tensor models from coordinates, forward and backward to the forces of
<dE/dv, v> or <dE/dA, A>, against the oracle's chain (GPU).  Tolerance as everywhere: 1e-11 in f64
(and df64), 2e-5 in f32, max-norm relative per output array."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import NP, TOL, lib, need_gpu, oracle_tables, rel

pytestmark = pytest.mark.gpu
DTYPES = [torch.float64, torch.float32]


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _cast(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a.astype(NP[dtype]))).cuda()


def _r(a, dtype):
    """The inputs as the GPU sees them (rounded to f32 for the f32 calls), for the oracle."""
    return a.astype(np.float32).astype(np.float64) if dtype == torch.float32 else a


@pytest.mark.parametrize("dtype", DTYPES, ids=["f64", "f32"])
@pytest.mark.parametrize("nloc,M1", [(1003, 100), (37, 1), (130, 37), (9, 256), (0, 100)])
def test_heads_against_oracle(dtype, nloc, M1):
    """v and A and their backward (dT overwritten, and added to a given dT with row 0 kept) on ragged
    atom counts and channel counts below, at and above a warp; a non-symmetric dE/dA."""
    dpc = lib()
    o = oracle.default()
    T = _r(W.normal(301, (nloc, 4, M1)), dtype)
    a = _r(W.normal(302, (nloc, M1)), dtype)
    dv = _r(W.normal(303, (nloc, 3)), dtype)
    dA = _r(W.normal(304, (nloc, 3, 3)), dtype)
    base = _r(W.normal(305, (nloc, 4, M1)), dtype)
    Tg, ag = _cast(T, dtype), _cast(a, dtype)
    v = dpc.dp_vector_head(Tg, ag)
    A = dpc.dp_tensor_head(Tg, ag)
    dTv, dav = dpc.dp_vector_head_grad(Tg, ag, _cast(dv, dtype))
    dTA, daA = dpc.dp_tensor_head_grad(Tg, ag, _cast(dA, dtype))
    acc = _cast(base, dtype)
    dpc.dp_tensor_head_grad(Tg, ag, _cast(dA, dtype), dT=acc, accumulate=True)
    none_dT, da_only = dpc.dp_vector_head_grad(Tg, ag, _cast(dv, dtype), want=("da",))
    acc_v = _cast(base, dtype)
    _, none_da = dpc.dp_vector_head_grad(Tg, ag, _cast(dv, dtype), dT=acc_v, accumulate=True, want=("dT",))
    assert none_dT is None and none_da is None
    torch.cuda.synchronize()
    if nloc == 0:
        assert v.shape == (0, 3) and A.shape == (0, 3, 3)
        return
    tol = TOL[dtype]
    assert rel(v.double().cpu().numpy(), o.vector_head(T, a)) <= tol
    Ao = o.tensor_head(T, a)
    Ag = A.double().cpu().numpy()
    assert rel(Ag, Ao) <= tol
    assert np.array_equal(Ag, np.transpose(Ag, (0, 2, 1)))  # mirrored from the six unique sums
    for (dTg, dag), (dTo, dao) in (((dTv, dav), o.vector_head_grad(T, a, dv)),
                                   ((dTA, daA), o.tensor_head_grad(T, a, dA))):
        assert rel(dTg.double().cpu().numpy(), dTo) <= tol
        assert not dTg[:, 0].any()
        assert rel(dag.double().cpu().numpy(), dao) <= tol
    assert torch.equal(da_only, dav)  # one output alone: the same bits
    for accg, (dTo, _) in ((acc, o.tensor_head_grad(T, a, dA)), (acc_v, o.vector_head_grad(T, a, dv))):
        got = accg.double().cpu().numpy()
        assert np.array_equal(got[:, 0], base[:, 0].astype(NP[dtype]).astype(np.float64))
        assert rel(got, base + dTo) <= tol


def test_head_refusals():
    """Shapes and types refused before any launch: a T that is not [nloc][4][M1], a of the wrong
    shape or type, accumulate without a dT."""
    dpc = lib()
    T = torch.zeros((5, 4, 8), dtype=torch.float64, device="cuda")
    a = torch.zeros((5, 8), dtype=torch.float64, device="cuda")
    with pytest.raises(ValueError):
        dpc.dp_vector_head(T[:, :3].contiguous(), a)
    with pytest.raises(ValueError):
        dpc.dp_tensor_head(T, a[:, :7].contiguous())
    with pytest.raises(TypeError):
        dpc.dp_vector_head(T, a.float())
    with pytest.raises(ValueError):
        dpc.dp_vector_head_grad(T, a, torch.zeros((5, 3), dtype=torch.float64, device="cuda"), accumulate=True)


ARITH = [("f64", torch.float64), ("f32", torch.float32), ("df64", torch.float64)]


@pytest.mark.parametrize("name,dtype", ARITH, ids=[a[0] for a in ARITH])
@pytest.mark.parametrize("hidden,nout,nat", [((64, 64, 64), 100, (70, 0, 33)), ((24,), 37, (65,)),
                                             ((48, 48), 3, (1, 40))], ids=["M1-out", "one-hidden", "three-out"])
def test_fitting_with_several_outputs(name, dtype, hidden, nout, nat):
    """A fitting net of nout outputs (the M1 weights of a head) and its backward weighted by
    g [nloc][nout], several centre types (one empty), against the oracle."""
    dpc = lib()
    ntypes = len(nat)
    widths = [70, *hidden, nout]
    params = W.net_params(311, widths, ntypes)
    ts = np.concatenate([[0], np.cumsum(nat)]).astype(np.int64)
    n = int(ts[-1])
    D = _r(W.normal(312, (n, 70)), dtype)
    g = _r(W.normal(313, (n, nout)), dtype)
    at = np.repeat(np.arange(ntypes), nat).astype(np.int32)
    arith = dpc.DF64 if name == "df64" else None
    p = _cast(_r(params, dtype), dtype)
    E, act = dpc.dp_fitting_fwd(p, widths, ts, _cast(D, dtype), arith=arith)
    dD = dpc.dp_fitting_grad(p, widths, ts, act, g=_cast(g, dtype), arith=arith)
    torch.cuda.synchronize()
    assert E.shape == (n, nout)
    Eo, dDo = oracle.default().fitting(_r(params, dtype), widths, D, at, g=g)
    tol = TOL[dtype]
    assert rel(E.double().cpu().numpy(), Eo) <= tol
    assert rel(dD.double().cpu().numpy(), dDo) <= tol
    with pytest.raises(dpc.DPError):  # several outputs need g
        dpc.dp_fitting_grad(p, widths, ts, act, arith=arith)
    if name == "f64":  # the net with its hidden layers on the tensor cores
        Et, actt = dpc.dp_fitting_fwd_tc_f64(p, widths, ts, _cast(D, dtype))
        dDt = dpc.dp_fitting_grad_tc_f64(p, widths, ts, actt, g=_cast(g, dtype))
        torch.cuda.synchronize()
        assert rel(Et.cpu().numpy(), Eo) <= tol and rel(dDt.cpu().numpy(), dDo) <= tol
        with pytest.raises(dpc.DPError):
            dpc.dp_fitting_grad_tc_f64(p, widths, ts, actt)


@pytest.mark.parametrize("head,tc_net", [("vector", False), ("tensor", False), ("vector", True)],
                         ids=["vector", "tensor", "vector-tc-net"])
def test_vector_and_tensor_models_from_coordinates(head, tc_net):
    """Coordinates -> s, R~ -> T, D (the tensor-core forward, D written by it) -> a = fitting net with
    M1 outputs -> v or A, and back for L = <dE/dv, v> or <dE/dA, A>: the head's dT added to the
    descriptor's (dE/da -> fitting backward -> dD -> dT), the tensor-core backward, forces and virial;
    every step on the GPU, against the oracle's chain; the folded forces sum to zero.  tc_net: the
    fitting net's hidden layers on the tensor cores."""
    dpc = lib()
    from test_gpu_env_force import _system
    w, coord, nlist, owner, env = _system("water", dict(seed=321, nmol=160), 0, None)
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    model = dpc.Model.compress(torch.from_numpy(w.params).cuda(), w.widths, info, torch.float64)
    plan = dpc.dp_tabulate_tc_plan_f64(model.table, info, w.nnei)
    widths = [w.M1 * w.M2, 48, 48, w.M1]
    fparams = W.net_params(322, widths, w.ntypes)
    ts = np.concatenate([[0], np.cumsum(np.bincount(w.atype, minlength=w.ntypes))]).astype(np.int64)
    shape = (w.nloc, 3) if head == "vector" else (w.nloc, 3, 3)
    dout = W.normal(323, shape)
    cg, ng, at = torch.from_numpy(coord).cuda(), torch.from_numpy(nlist).cuda(), torch.from_numpy(w.atype).cuda()
    ei = dpc.env_info(*env)
    s, Rt, nvalid = dpc.dp_env_mat(cg, ng, w.sel, ei)
    T, D = dpc.dp_tabulate_fusion_fwd_tc_f64(plan, info, s, Rt, nvalid, at, w.sel, M2=w.M2)
    fp = torch.from_numpy(fparams).cuda()
    fit_fwd = dpc.dp_fitting_fwd_tc_f64 if tc_net else dpc.dp_fitting_fwd
    fit_grad = dpc.dp_fitting_grad_tc_f64 if tc_net else dpc.dp_fitting_grad
    a, act = fit_fwd(fp, widths, ts, D)
    fwd_head = dpc.dp_vector_head if head == "vector" else dpc.dp_tensor_head
    grad_head = dpc.dp_vector_head_grad if head == "vector" else dpc.dp_tensor_head_grad
    out = fwd_head(T, a)
    dT0, da = grad_head(T, a, torch.from_numpy(dout).cuda())
    dD = fit_grad(fp, widths, ts, act, g=da)
    dT = dpc.dp_descriptor_contract_grad(T, dD.reshape(D.shape))
    dT_desc = dT.clone()
    grad_head(T, a, torch.from_numpy(dout).cuda(), dT=dT, accumulate=True)
    ds, dRt = dpc.dp_tabulate_fusion_grad_tc_f64(plan, info, s, Rt, nvalid, at, w.sel, dT)
    F, Wv = dpc.dp_force_virial(cg, ng, ei, ds, dRt)
    torch.cuda.synchronize()
    o = oracle.default()
    oi, tabs = oracle_tables(w, torch.float64)
    so, Rto = o.env_mat(coord, nlist, *env)
    To = o.fwd(tabs, oi, so, Rto, w.nvalid, w.atype, w.sel)
    Do = o.descriptor(To, w.M2)
    ao = o.fitting(fparams, widths, Do.reshape(w.nloc, -1), w.atype, grad=False)
    if head == "vector":
        outo = o.vector_head(To, ao)
        dTho, dao = o.vector_head_grad(To, ao, dout)
    else:
        outo = o.tensor_head(To, ao)
        dTho, dao = o.tensor_head_grad(To, ao, dout)
    _, dDo = o.fitting(fparams, widths, Do.reshape(w.nloc, -1), w.atype, g=dao)
    dTo = o.descriptor_grad(To, dDo.reshape(Do.shape)) + dTho
    dso, dRo = o.grad(tabs, oi, so, Rto, w.nvalid, w.atype, w.sel, dTo)
    Fo, Wo = o.force_virial(coord, nlist, env[0], env[1], dso, dRo, env[2], env[3])
    for got, ref, k in ((out, outo, "head"), (a, ao, "a"), (da, dao, "da"), (dT0, dTho, "dT of the head"),
                        (dT, dTo, "dT"), (F, Fo, "F"), (Wv, Wo, "virial")):
        assert rel(got.cpu().numpy(), ref) <= 1e-11, (k, rel(got.cpu().numpy(), ref))
    assert torch.equal(dT[:, 0], dT_desc[:, 0])  # the head adds nothing to row 0
    folded = np.zeros((w.nloc, 3))
    np.add.at(folded, owner, F.cpu().numpy())
    assert np.abs(folded.sum(axis=0)).max() <= 1e-9 * np.abs(folded).max()


def test_fitting_noalloc_with_several_outputs():
    """dp_fitting_grad_noalloc_f64 on a net of several outputs (its scratch from the library's fixed
    array) gives the bits of dp_fitting_grad_f64 with a work buffer; without g it is refused."""
    dpc = lib()
    widths = [40, 32, 32, 12]
    params = W.net_params(331, widths, 2)
    ts = np.array([0, 30, 75], dtype=np.int64)
    D = W.normal(332, (75, 40))
    g = W.normal(333, (75, 12))
    p = torch.from_numpy(params).cuda()
    E, act = dpc.dp_fitting_fwd(p, widths, ts, torch.from_numpy(D).cuda())
    gd = torch.from_numpy(g).cuda()
    a = dpc.dp_fitting_grad(p, widths, ts, act, g=gd)
    b = dpc.dp_fitting_grad_noalloc_f64(p, widths, ts, act, g=gd)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    with pytest.raises(dpc.DPError):
        dpc.dp_fitting_grad_noalloc_f64(p, widths, ts, act)
