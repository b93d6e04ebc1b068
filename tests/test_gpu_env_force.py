"""Environment-matrix front end and force/virial back end on the GPU vs the oracle (GPU).

Inputs are the workloads' own positions and formatted neighbour lists, with periodic images
turned into extra coordinates (workloads.ghost_system); the oracle runs on the same arrays
(f32: on the f32-rounded arrays, in f64 arithmetic).
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import NP, TOL, lib, need_gpu, oracle_tables, product_model, rel

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _r(a, dtype):
    return a.astype(np.float32).astype(np.float64) if dtype == torch.float32 else a


SYSTEMS = [
    ("cu", dict(seed=41, cells=(6, 6, 6), sel=256, fill=0.8), 0, None),
    ("cu", dict(seed=42, cells=(6, 6, 6), sel=256, fill=0.8), 1, None),
    ("water", dict(seed=43, nmol=256), 0, None),
    ("water", dict(seed=44, nmol=256), 1, (0.05, 0.1, 0.2)),
]


def _system(name, kw, kind, norm):
    w = (W.cu if name == "cu" else W.water)(widths=(1, 8, 16, 32), M2=8, **kw)
    coord, nlist, owner = W.ghost_system(w)
    return w, coord, nlist, owner, (w.env["rcs"], w.env["rc"], kind, norm)


@pytest.mark.parametrize("name,kw,kind,norm", SYSTEMS, ids=[f"{s[0]}-k{s[2]}-n{s[3] is not None}" for s in SYSTEMS])
@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_env_mat(name, kw, kind, norm, dtype):
    """s, R~ and the per-segment counts from coordinates + neighbour list."""
    dpc = lib()
    w, coord, nlist, _, env = _system(name, kw, kind, norm)
    c = _r(coord, dtype)
    s, Rt, nvalid = dpc.dp_env_mat(torch.from_numpy(c.astype(NP[dtype])).cuda(), torch.from_numpy(nlist).cuda(),
                                   w.sel, dpc.env_info(*env))
    torch.cuda.synchronize()
    so, Rto = oracle.default().env_mat(c, nlist, *env)
    assert np.array_equal(nvalid.cpu().numpy(), w.nvalid)
    assert rel(s.double().cpu().numpy(), so) <= TOL[dtype]
    assert rel(Rt.double().cpu().numpy(), Rto) <= TOL[dtype]
    pad = nlist < 0
    assert not s.cpu().numpy()[pad].any() and not Rt.cpu().numpy()[pad].any()


@pytest.mark.parametrize("name,kw,kind,norm", SYSTEMS, ids=[f"{s[0]}-k{s[2]}-n{s[3] is not None}" for s in SYSTEMS])
@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_force_virial(name, kw, kind, norm, dtype):
    """F on every coordinate row and the virial from given dE/ds, dE/dR~ (stale outputs overwritten)."""
    dpc = lib()
    w, coord, nlist, _, env = _system(name, kw, kind, norm)
    c = _r(coord, dtype)
    ds = _r(W.normal(7, nlist.shape), dtype)
    dRt = _r(W.normal(8, nlist.shape + (4,)), dtype)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a.astype(NP[dtype]))).cuda()  # noqa: E731
    stale = (torch.full((coord.shape[0], 3), 5.0, dtype=dtype, device="cuda"),
             torch.full((3, 3), 5.0, dtype=dtype, device="cuda"))
    F, Wv = dpc.dp_force_virial(dev(c), torch.from_numpy(nlist).cuda(), dpc.env_info(*env), dev(ds), dev(dRt),
                                out=stale)
    torch.cuda.synchronize()
    Fo, Wo = oracle.default().force_virial(c, nlist, env[0], env[1], ds, dRt, env[2], env[3])
    assert rel(F.double().cpu().numpy(), Fo) <= TOL[dtype]
    assert rel(Wv.double().cpu().numpy(), Wo) <= TOL[dtype]


@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
@pytest.mark.parametrize("moments", [False, True])
def test_forces_through_the_whole_chain(dtype, moments):
    """coordinates -> rows -> fused forward -> D -> dE/dD -> dE/dT -> dE/ds, dE/dR~ -> forces, virial, all on
    the GPU, against the oracle's chain; the folded forces of the periodic system sum to zero."""
    dpc = lib()
    w, coord, nlist, owner, env = _system("water", dict(seed=45, nmol=256), 1, None)
    c = _r(coord, dtype)
    model = product_model(w, dtype)
    cg = torch.from_numpy(c.astype(NP[dtype])).cuda()
    ng = torch.from_numpy(nlist).cuda()
    at = torch.from_numpy(w.atype).cuda()
    ei = dpc.env_info(*env)
    dD = _r(W.normal(46, (w.nloc, w.M1, w.M2)), dtype)
    fwd = dpc.dp_tabulate_fusion_fwd_moments if moments else dpc.dp_tabulate_fusion_fwd
    grad = dpc.dp_tabulate_fusion_grad_moments if moments else dpc.dp_tabulate_fusion_grad
    s, Rt, nvalid = dpc.dp_env_mat(cg, ng, w.sel, ei)
    T = fwd(model.table, model.info, s, Rt, nvalid, at, w.sel)
    dT = dpc.dp_descriptor_contract_grad(T, torch.from_numpy(dD.astype(NP[dtype])).cuda())
    ds, dRt = grad(model.table, model.info, s, Rt, nvalid, at, w.sel, dT)
    F, Wv = dpc.dp_force_virial(cg, ng, ei, ds, dRt)
    torch.cuda.synchronize()
    o = oracle.default()
    info, tabs = oracle_tables(w, dtype)
    so, Rto = o.env_mat(c, nlist, *env)
    To = o.fwd(tabs, info, so, Rto, w.nvalid, w.atype, w.sel)
    dso, dRo = o.grad(tabs, info, so, Rto, w.nvalid, w.atype, w.sel, o.descriptor_grad(To, dD))
    Fo, Wo = o.force_virial(c, nlist, env[0], env[1], dso, dRo, env[2], env[3])
    tol = TOL[dtype] * (1 if dtype == torch.float64 else 5)
    assert rel(F.double().cpu().numpy(), Fo) <= tol
    assert rel(Wv.double().cpu().numpy(), Wo) <= tol
    folded = np.zeros((w.nloc, 3))
    np.add.at(folded, owner, F.double().cpu().numpy())
    assert np.abs(folded.sum(axis=0)).max() <= 1e-9 * np.abs(folded).max() * (1 if dtype == torch.float64 else 1e4)


def test_env_force_edges():
    """nloc = 0; every row padding; a neighbour exactly at rc (s = 0 and no force); both dtypes."""
    dpc = lib()
    ei = dpc.env_info(1.0, 3.0, kind=1)
    for dt in (torch.float64, torch.float32):
        coord = torch.tensor([[0.0, 0.0, 0.0], [3.0, 0.0, 0.0], [3.0, 2.0, 0.0]], dtype=dt, device="cuda")
        s, Rt, nv = dpc.dp_env_mat(coord, torch.empty((0, 4), dtype=torch.int32, device="cuda"), [4], ei)
        assert s.shape == (0, 4) and nv.shape == (0, 1)
        nl = torch.tensor([[-1, -1, -1, -1], [0, 2, -1, -1]], dtype=torch.int32, device="cuda")
        s, Rt, nv = dpc.dp_env_mat(coord, nl, [4], ei)
        torch.cuda.synchronize()
        assert nv.cpu().tolist() == [[0], [2]]
        assert not s[0].abs().max().item() and s[1, 0].item() == 0.0  # r = rc: outside
        assert s[1, 1].item() == 0.25  # r = 2: u = 1/2, w = 1/2 exactly
        F, Wv = dpc.dp_force_virial(coord, nl, ei, torch.ones((2, 4), dtype=dt, device="cuda"),
                                    torch.ones((2, 4, 4), dtype=dt, device="cuda"))
        torch.cuda.synchronize()
        Fo, Wo = oracle.default().force_virial(coord.double().cpu().numpy(), nl.cpu().numpy(), 1.0, 3.0,
                                               np.ones((2, 4)), np.ones((2, 4, 4)), 1)
        assert rel(F.double().cpu().numpy(), Fo) <= TOL[dt] and rel(Wv.double().cpu().numpy(), Wo) <= TOL[dt]
        F0, W0 = dpc.dp_force_virial(coord, torch.empty((0, 4), dtype=torch.int32, device="cuda"), ei,
                                     torch.empty((0, 4), dtype=dt, device="cuda"),
                                     torch.empty((0, 4, 4), dtype=dt, device="cuda"))
        torch.cuda.synchronize()
        assert not F0.abs().max().item() and not W0.abs().max().item()


@pytest.mark.parametrize("name,kind,reuse", [("water", 1, True), ("water", 0, False), ("cu", 1, True)])
def test_fused_env_chain_on_the_tensor_cores(name, kind, reuse):
    """The fused front and back end of the tensor-core path (dp_tabulate_fusion_env_{fwd,grad}_tc_f64: rows formed
    from coordinates, forces added in the rows kernel) against the same chain unfused (dp_env_mat ->
    dp_tabulate_fusion_fwd_tc_f64 -> dp_descriptor_contract_grad -> dp_tabulate_fusion_grad_tc_f64 ->
    dp_force_virial): T, D and nvalid bit for bit (the same rows), F and the virial to 1e-12 (the order of
    the atomic additions), and the oracle's chain within the f64 tolerance; the folded forces sum to zero."""
    dpc = lib()
    kw = dict(seed=47, nmol=256) if name == "water" else dict(seed=48, cells=(6, 6, 6), sel=256, fill=0.8)
    w, coord, nlist, owner, env = _system(name, kw, kind, None)
    model = product_model(w, torch.float64)
    cg = torch.from_numpy(coord).cuda()
    ng = torch.from_numpy(nlist).cuda()
    at = torch.from_numpy(w.atype).cuda()
    ei = dpc.env_info(*env)
    dD = torch.from_numpy(W.normal(49, (w.nloc, w.M1, w.M2))).cuda()
    plan = dpc.dp_tabulate_tc_plan_f64(model.table, model.info, w.nnei)
    work = torch.empty((dpc.dp_tabulate_tc_work_bytes(model.info, w.nloc, w.nnei, w.ntypes, w.M1),),
                       dtype=torch.uint8, device="cuda")
    # unfused
    s, Rt, nv = dpc.dp_env_mat(cg, ng, w.sel, ei)
    T0, D0 = dpc.dp_tabulate_fusion_fwd_tc_f64(plan, model.info, s, Rt, nv, at, w.sel, work=work, M2=w.M2)
    dT0 = dpc.dp_descriptor_contract_grad(T0, dD)
    ds, dRt = dpc.dp_tabulate_fusion_grad_tc_f64(plan, model.info, s, Rt, nv, at, w.sel, dT0, work=work,
                                                 flags=dpc.DP_TC_REUSE_RUNS)
    F0, W0 = dpc.dp_force_virial(cg, ng, ei, ds, dRt)
    # fused
    T1, D1, nv1 = dpc.dp_tabulate_fusion_env_fwd_tc_f64(plan, model.info, cg, ng, w.sel, ei, at, work=work, M2=w.M2)
    dT1 = dpc.dp_descriptor_contract_grad(T1, dD)
    F1, W1 = dpc.dp_tabulate_fusion_env_grad_tc_f64(plan, model.info, cg, ng, w.sel, ei, at, dT1, work=work,
                                                    flags=dpc.DP_TC_REUSE_RUNS if reuse else 0)
    torch.cuda.synchronize()
    assert torch.equal(nv1, nv) and torch.equal(T1, T0) and torch.equal(D1, D0)
    assert rel(F1.cpu().numpy(), F0.cpu().numpy()) <= 1e-12 and rel(W1.cpu().numpy(), W0.cpu().numpy()) <= 1e-12
    o = oracle.default()
    info, tabs = oracle_tables(w, torch.float64)
    so, Rto = o.env_mat(coord, nlist, *env)
    To = o.fwd(tabs, info, so, Rto, w.nvalid, w.atype, w.sel)
    dso, dRo = o.grad(tabs, info, so, Rto, w.nvalid, w.atype, w.sel, o.descriptor_grad(To, dD.cpu().numpy()))
    Fo, Wo = o.force_virial(coord, nlist, env[0], env[1], dso, dRo, env[2], env[3])
    assert rel(T1.cpu().numpy(), To) <= TOL[torch.float64]
    assert rel(F1.cpu().numpy(), Fo) <= TOL[torch.float64] and rel(W1.cpu().numpy(), Wo) <= TOL[torch.float64]
    folded = np.zeros((w.nloc, 3))
    np.add.at(folded, owner, F1.cpu().numpy())
    assert np.abs(folded.sum(axis=0)).max() <= 1e-9 * np.abs(folded).max()


def test_fused_env_edges():
    """The fused calls on nloc = 0 (F and the virial still zeroed) and on atoms whose rows are all padding
    or sit at rc (s = 0, no force), against the unfused chain."""
    dpc = lib()
    ei = dpc.env_info(1.0, 3.0, kind=1)
    w = W.tiny(seed=50, nloc=3, nreal=4, sel=4, widths=(1, 4, 8), M2=2)
    model = product_model(w, torch.float64)
    plan = dpc.dp_tabulate_tc_plan_f64(model.table, model.info, 4)
    coord = torch.tensor([[0.0, 0.0, 0.0], [3.0, 0.0, 0.0], [3.0, 2.0, 0.0], [1.5, 0.5, 0.2]], dtype=torch.float64,
                         device="cuda")
    nl = torch.tensor([[-1, -1, -1, -1], [0, 2, 3, -1], [1, 3, -1, -1]], dtype=torch.int32, device="cuda")
    T, D, nv = dpc.dp_tabulate_fusion_env_fwd_tc_f64(plan, model.info, coord, nl, [4], ei, M2=2)
    dT = torch.ones_like(T)
    F, Wv = dpc.dp_tabulate_fusion_env_grad_tc_f64(plan, model.info, coord, nl, [4], ei, None, dT)
    s, Rt, nv0 = dpc.dp_env_mat(coord, nl, [4], ei)
    T0 = dpc.dp_tabulate_fusion_fwd_tc_f64(plan, model.info, s, Rt, nv0, None, [4])
    ds, dRt = dpc.dp_tabulate_fusion_grad_tc_f64(plan, model.info, s, Rt, nv0, None, [4], dT)
    F0, W0 = dpc.dp_force_virial(coord, nl, ei, ds, dRt)
    torch.cuda.synchronize()
    assert nv.cpu().tolist() == [[0], [3], [2]] and torch.equal(nv, nv0) and torch.equal(T, T0)
    assert not T[0].abs().max().item()
    assert rel(F.cpu().numpy(), F0.cpu().numpy()) <= 1e-12 and rel(Wv.cpu().numpy(), W0.cpu().numpy()) <= 1e-12
    e3 = torch.empty((0, 4), dtype=torch.int32, device="cuda")
    Fz, Wz = dpc.dp_tabulate_fusion_env_grad_tc_f64(plan, model.info, coord, e3, [4], ei, None,
                                                    torch.empty((0, 4, w.M1), dtype=torch.float64, device="cuda"),
                                                    out=(torch.full((4, 3), 7.0, dtype=torch.float64, device="cuda"),
                                                         torch.full((3, 3), 7.0, dtype=torch.float64, device="cuda")))
    torch.cuda.synchronize()
    assert not Fz.abs().max().item() and not Wz.abs().max().item()
