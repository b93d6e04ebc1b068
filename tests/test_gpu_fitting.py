"""Fitting net (D_i -> E_i) and its backward on the GPU vs the oracle, and the whole model from
coordinates to energy and forces (GPU).  Tolerance as everywhere: 1e-11 in f64 and df64, 2e-5 in f32
(max-norm relative per output array)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import NP, TOL, lib, need_gpu, oracle_tables, rel

pytestmark = pytest.mark.gpu
ARITH = [("f64", torch.float64), ("f32", torch.float32), ("df64", torch.float64)]


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _tol(name):
    return TOL[torch.float32] if name == "f32" else TOL[torch.float64]


def _run(dpc, name, dtype, params, widths, ts, D, g=None):
    arith = dpc.DF64 if name == "df64" else None
    cast = lambda a: torch.from_numpy(np.ascontiguousarray(a.astype(NP[dtype]))).cuda()  # noqa: E731
    p = cast(params)
    E, act = dpc.dp_fitting_fwd(p, widths, ts, cast(D), arith=arith)
    dD = dpc.dp_fitting_grad(p, widths, ts, act, g=None if g is None else cast(g), arith=arith)
    torch.cuda.synchronize()
    return E.double().cpu().numpy(), dD.double().cpu().numpy()


def _r(a, name):
    return a.astype(np.float32).astype(np.float64) if name == "f32" else a


@pytest.mark.parametrize("name,dtype", ARITH, ids=[a[0] for a in ARITH])
@pytest.mark.parametrize("hidden,nat,ntypes", [((240, 240, 240), (300, 0, 77), 3), ((37, 37, 50), (65,), 1),
                                               ((24,), (33, 31), 2), ((8, 8), (129, 1), 2)],
                         ids=["paper", "ragged", "one-hidden", "tiny-tiles"])
def test_fitting_against_oracle(name, dtype, hidden, nat, ntypes):
    """E and dE/dD for several centre types (one of them empty), widths that are not multiples of the
    tiles, a single hidden layer (no scratch), upstream weights g."""
    dpc = lib()
    K = 1600 if hidden == (240, 240, 240) else 70
    widths, params = W.fitting_net(7, K, hidden, ntypes)
    ts = np.concatenate([[0], np.cumsum(nat)]).astype(np.int64)
    n = int(ts[-1])
    D = _r(W.normal(8, (n, K), 0.0, 0.3), name)
    g = _r(W.normal(9, (n,)), name)
    at = np.repeat(np.arange(ntypes), nat).astype(np.int32)
    E, dD = _run(dpc, name, dtype, params, widths, ts, D, g)
    Eo, dDo = oracle.default().fitting(_r(params, name), widths, D, at, g=g)
    assert rel(E, Eo) <= _tol(name), rel(E, Eo)
    assert rel(dD, dDo) <= _tol(name), rel(dD, dDo)


def test_fitting_skip_on_the_input_layer_and_errors():
    """A first hidden layer as wide as D (its skip adds D itself); empty input; bad shapes rejected."""
    dpc = lib()
    widths, params = W.fitting_net(11, 48, (48, 48), 1)
    D = W.normal(12, (70, 48))
    E, dD = _run(dpc, "f64", torch.float64, params, widths, [0, 70], D)
    Eo, dDo = oracle.default().fitting(params, widths, D)
    assert rel(E, Eo) <= 1e-11 and rel(dD, dDo) <= 1e-11
    p = torch.from_numpy(params).cuda()
    E0, act0 = dpc.dp_fitting_fwd(p, widths, [0, 0], torch.empty((0, 48), dtype=torch.float64, device="cuda"))
    assert E0.shape == (0,)
    with pytest.raises((ValueError, dpc.DPError)):
        dpc.dp_fitting_fwd(p, widths[:-1] + [2], [0, 70], torch.from_numpy(D).cuda())
    with pytest.raises(ValueError):
        dpc.dp_fitting_fwd(p, widths, [0, 70, 71], torch.from_numpy(D).cuda())


@pytest.mark.parametrize("arith", ["f64", "df64", "f64-tc"])
def test_energy_and_forces_of_the_whole_model(arith):
    """Coordinates -> s, R~ -> T -> D -> E_i (fitting net) and back: dE/dD -> dE/dT -> dE/ds, dE/dR~ ->
    forces and virial, every step on the GPU, against the oracle's chain; the folded forces sum to zero.
    f64-tc: the fitting net's GEMMs on the tensor cores (dp_fitting_*_tc_f64)."""
    dpc = lib()
    from test_gpu_env_force import _system
    w, coord, nlist, owner, env = _system("water", dict(seed=47, nmol=128), 0, None)
    df = arith == "df64"
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    model = dpc.Model.compress(torch.from_numpy(w.params).cuda(), w.widths, info, dpc.DF64 if df else torch.float64)
    widths, fparams = W.fitting_net(13, w.M1 * w.M2, (64, 64, 64), w.ntypes)
    ts = np.concatenate([[0], np.cumsum(np.bincount(w.atype, minlength=w.ntypes))]).astype(np.int64)
    a = dpc.DF64 if df else None
    cg, ng, at = torch.from_numpy(coord).cuda(), torch.from_numpy(nlist).cuda(), torch.from_numpy(w.atype).cuda()
    ei = dpc.env_info(*env)
    fwd = dpc.dp_tabulate_fusion_fwd_moments
    grad = dpc.dp_tabulate_fusion_grad_moments
    s, Rt, nvalid = dpc.dp_env_mat(cg, ng, w.sel, ei, arith=a)
    T = fwd(model.table, model.info, s, Rt, nvalid, at, w.sel)
    D = dpc.dp_descriptor_contract(T, w.M2, arith=a)
    fp = torch.from_numpy(fparams).cuda()
    if arith == "f64-tc":
        E, act = dpc.dp_fitting_fwd_tc_f64(fp, widths, ts, D)
        dD = dpc.dp_fitting_grad_tc_f64(fp, widths, ts, act)
    else:
        E, act = dpc.dp_fitting_fwd(fp, widths, ts, D, arith=a)
        dD = dpc.dp_fitting_grad(fp, widths, ts, act, arith=a)
    dT = dpc.dp_descriptor_contract_grad(T, dD.reshape(D.shape), arith=a)
    ds, dRt = grad(model.table, model.info, s, Rt, nvalid, at, w.sel, dT)
    F, Wv = dpc.dp_force_virial(cg, ng, ei, ds, dRt, arith=a)
    torch.cuda.synchronize()
    o = oracle.default()
    oi, tabs = oracle_tables(w, torch.float64)
    so, Rto = o.env_mat(coord, nlist, *env)
    To = o.fwd(tabs, oi, so, Rto, w.nvalid, w.atype, w.sel)
    Do = o.descriptor(To, w.M2)
    Eo, dDo = o.fitting(fparams, widths, Do.reshape(w.nloc, -1), w.atype)
    dso, dRo = o.grad(tabs, oi, so, Rto, w.nvalid, w.atype, w.sel, o.descriptor_grad(To, dDo.reshape(Do.shape)))
    Fo, Wo = o.force_virial(coord, nlist, env[0], env[1], dso, dRo, env[2], env[3])
    for got, ref in ((E, Eo), (F, Fo), (Wv, Wo)):
        assert rel(got.cpu().numpy(), ref) <= 1e-11, rel(got.cpu().numpy(), ref)
    assert abs(E.sum().item() - Eo.sum()) <= 1e-11 * np.abs(Eo).sum()
    folded = np.zeros((w.nloc, 3))
    np.add.at(folded, owner, F.cpu().numpy())
    assert np.abs(folded.sum(axis=0)).max() <= 1e-9 * np.abs(folded).max()
