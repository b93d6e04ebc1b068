"""df64 (double-float) variant of the moment path vs the oracle (GPU).

The df64 calls take and return double arrays and must meet the f64 tolerance (1e-11, max-norm
relative per output array) against the oracle, which runs in double on the same inputs.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import TOL, assert_parity, lib, need_gpu, oracle_tables, product_model, rel, run_oracle, to_dev, \
    workload

pytestmark = pytest.mark.gpu
F64 = torch.float64


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def df64_model(w):
    dpc = lib()
    info = dpc.dp_table_info_make(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    return dpc.Model.compress(torch.from_numpy(w.params).cuda(), w.widths, info, dpc.DF64)


def run_df64(w, model=None, x=None, out=None):
    dpc = lib()
    model = model or df64_model(w)
    x = x or to_dev(w, F64)
    T = dpc.dp_tabulate_fusion_fwd_moments_df64(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"],
                                                w.sel, out=None if out is None else out[0])
    D = dpc.dp_descriptor_contract_df64(T, w.M2)
    ds, dRt = dpc.dp_tabulate_fusion_grad_moments_df64(model.table, model.info, x["s"], x["Rt"], x["nvalid"],
                                                       x["atype"], w.sel, x["dT"],
                                                       out=None if out is None else out[1:])
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in dict(T=T, D=D, ds=ds, dRt=dRt).items()}


def test_df64_table_splits_the_f64_table():
    """Each df64 coefficient is the f64 coefficient split into a float and the float rounding of the rest:
    hi + lo reproduces it to 2^-48 relative, and hi is the float rounding of the coefficient."""
    dpc = lib()
    w = workload("water", nmol=64, sel=(40, 80))
    info = dpc.dp_table_info_make(w.s_min, w.s_max)
    y, dy, d2y = dpc.dp_embedding_net_nodes(torch.from_numpy(w.params).cuda(), w.widths, info)
    t64 = dpc.dp_table_build(y, dy, d2y, info, F64).cpu().numpy()
    tdf = dpc.dp_table_build_df64(y, dy, d2y, info).cpu().numpy()
    assert tdf.shape == t64.shape[:-1] + (4,)
    hi = tdf[..., 0::2].astype(np.float64)
    lo = tdf[..., 1::2].astype(np.float64)
    assert np.array_equal(tdf[..., 0::2], t64.astype(np.float32))
    err = np.abs(hi + lo - t64)
    assert np.all(err <= 2.0 ** -48 * np.abs(t64) + 1e-300)


DF64_CASES = [
    ("tiny", {}, None), ("water", dict(nmol=256), None), ("cu85", dict(cells=(6, 6, 6)), None),
    ("cugeo", dict(cells=(6, 6, 6)), None), ("alcumg", dict(pad=0.1, cells=(6, 6, 6)), None),
    ("cu85", {}, None), ("alcumg", dict(pad=0.3), 384),
]


@pytest.mark.parametrize("name,kw,nsample", DF64_CASES, ids=[f"{c[0]}-{c[1]}" for c in DF64_CASES])
def test_df64_parity(name, kw, nsample):
    """T, D, ds and dR~ of the df64 path against the oracle (f64 tolerance), and against the f64 moment path."""
    dpc = lib()
    w = workload(name, **kw)
    x = to_dev(w, F64)
    got = run_df64(w, x=x)
    atoms = None
    if nsample:
        atoms = np.sort(np.random.default_rng(5).choice(w.nloc, nsample, replace=False))
    ref = run_oracle(w, F64, atoms=atoms)
    errs = assert_parity(got, ref, F64, atoms=atoms)
    print(f"df64 {name} {kw}: max-norm relative error vs the oracle {errs}")
    m64 = product_model(w, F64)
    T64 = dpc.dp_tabulate_fusion_fwd_moments(m64.table, m64.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    ds64, dR64 = dpc.dp_tabulate_fusion_grad_moments(m64.table, m64.info, x["s"], x["Rt"], x["nvalid"], x["atype"],
                                                     w.sel, x["dT"])
    torch.cuda.synchronize()
    for k, v in dict(T=T64, ds=ds64, dRt=dR64).items():
        assert rel(got[k], v.cpu().numpy()) <= TOL[F64]


@pytest.mark.parametrize("M1,widths", [(1, (1, 1)), (37, (1, 5, 37)), (64, (1, 16, 32, 64)), (200, (1, 50, 100, 200)),
                                       (256, (1, 64, 128, 256))])
def test_df64_shapes_clamps_nan(M1, widths):
    """Every channel-round shape with long runs, inputs past the coarse segment, below the table and NaN."""
    w = W.tiny(seed=95 + M1, nloc=11, nreal=27, sel=30, widths=widths, M2=1, rmin=2.6, rmax=3.0)
    s = w.s.copy()
    s[0, 0], s[1, 2], s[2, 1] = w.s_max * 7.0, w.s_min - 1.0, np.nan
    w2 = W.Workload(**{**w.__dict__, "s": s})
    got = run_df64(w2)
    ref = run_oracle(w2, F64)
    for k in ("T", "ds", "dRt", "D"):
        nan = np.isnan(ref[k])
        assert np.array_equal(np.isnan(got[k]), nan), k
        got[k][nan] = ref[k][nan] = 0.0
    assert_parity(got, ref, F64)


def test_df64_outputs_overwritten_and_empty():
    """Stale outputs are overwritten (padding rows zeroed); atoms without neighbours; nloc = 0."""
    dpc = lib()
    w = W.tiny(seed=7, nloc=5, nreal=5, sel=8)
    nv = w.nvalid.copy()
    nv[1] = 0
    w2 = W.Workload(**{**w.__dict__, "nvalid": nv})
    stale = (torch.full((w.nloc, 4, w.M1), np.nan, dtype=F64, device="cuda"),
             torch.full((w.nloc, w.nnei), 7.0, dtype=F64, device="cuda"),
             torch.full((w.nloc, w.nnei, 4), -3.0, dtype=F64, device="cuda"))
    got = run_df64(w2, out=stale)
    assert_parity(got, run_oracle(w2, F64), F64)
    assert not np.abs(got["T"][1]).max() and not np.abs(got["ds"][1]).max()
    model = df64_model(w)
    e = torch.empty((0, w.nnei), dtype=F64, device="cuda")
    T = dpc.dp_tabulate_fusion_fwd_moments_df64(model.table, model.info, e, e.reshape(0, w.nnei, 1).expand(0, w.nnei, 4)
                                                .contiguous(), None, None, w.sel)
    assert T.shape == (0, 4, w.M1)


def test_df64_descriptor_grad():
    """dE/dT from dE/dD in df64 against the oracle, and the chain dD -> dT -> ds, dR~."""
    dpc = lib()
    w = workload("water", nmol=128)
    o = oracle.default()
    x = to_dev(w, F64)
    model = df64_model(w)
    dD = W.normal(71, (w.nloc, w.M1, w.M2))
    T = dpc.dp_tabulate_fusion_fwd_moments_df64(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"],
                                                w.sel)
    dT = dpc.dp_descriptor_contract_grad_df64(T, torch.from_numpy(dD).cuda())
    ds, dRt = dpc.dp_tabulate_fusion_grad_moments_df64(model.table, model.info, x["s"], x["Rt"], x["nvalid"],
                                                       x["atype"], w.sel, dT)
    torch.cuda.synchronize()
    info, tabs = oracle_tables(w, F64)
    To = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    dTo = o.descriptor_grad(To, dD)
    dso, dRo = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, dTo)
    assert rel(dT.cpu().numpy(), dTo) <= TOL[F64]
    assert rel(ds.cpu().numpy(), dso) <= TOL[F64]
    assert rel(dRt.cpu().numpy(), dRo) <= TOL[F64]


def test_df64_water_large_sampled():
    """1,048,576 atoms in the benchmark's launch configuration; 256 sampled atoms against the oracle."""
    w = workload("water_large")
    atoms = np.concatenate([np.arange(64), np.sort(np.random.default_rng(6).choice(w.nloc, 128, replace=False)),
                            np.arange(w.nloc - 64, w.nloc)])
    got = run_df64(w)
    ref = run_oracle(w, F64, atoms=atoms)
    assert_parity(got, ref, F64, atoms=atoms)


# ------------------------------------------------------------- front and back end in df64
from test_gpu_env_force import SYSTEMS, _system  # noqa: E402


@pytest.mark.parametrize("name,kw,kind,norm", SYSTEMS, ids=[f"{s[0]}-k{s[2]}-n{s[3] is not None}" for s in SYSTEMS])
def test_df64_env_mat_and_forces(name, kw, kind, norm):
    """s, R~, counts, forces and virial in df64 against the oracle (both switches, normalised or not)."""
    dpc = lib()
    w, coord, nlist, _, env = _system(name, kw, kind, norm)
    cg, ng = torch.from_numpy(coord).cuda(), torch.from_numpy(nlist).cuda()
    ei = dpc.env_info(*env)
    s, Rt, nvalid = dpc.dp_env_mat_df64(cg, ng, w.sel, ei)
    ds = W.normal(7, nlist.shape)
    dRt = W.normal(8, nlist.shape + (4,))
    stale = (torch.full((coord.shape[0], 3), 5.0, dtype=F64, device="cuda"),
             torch.full((3, 3), 5.0, dtype=F64, device="cuda"))
    F, Wv = dpc.dp_force_virial_df64(cg, ng, ei, torch.from_numpy(ds).cuda(), torch.from_numpy(dRt).cuda(), out=stale)
    torch.cuda.synchronize()
    o = oracle.default()
    so, Rto = o.env_mat(coord, nlist, *env)
    Fo, Wo = o.force_virial(coord, nlist, env[0], env[1], ds, dRt, env[2], env[3])
    assert np.array_equal(nvalid.cpu().numpy(), w.nvalid)
    errs = {k: rel(g, r) for k, g, r in (("s", s.cpu().numpy(), so), ("Rt", Rt.cpu().numpy(), Rto),
                                          ("F", F.cpu().numpy(), Fo), ("virial", Wv.cpu().numpy(), Wo))}
    print(f"df64 env/force {name} kind={kind} norm={norm is not None}: {errs}")
    assert all(e <= TOL[F64] for e in errs.values()), errs
    assert not s.cpu().numpy()[nlist < 0].any()


def test_df64_forces_through_the_whole_chain():
    """coordinates -> rows -> T -> D -> dE/dT -> dE/ds, dE/dR~ -> forces, virial, every kernel in df64,
    against the oracle's chain; the folded forces of the periodic system sum to zero."""
    dpc = lib()
    w, coord, nlist, owner, env = _system("water", dict(seed=45, nmol=256), 1, None)
    model = df64_model(w)
    cg, ng, at = torch.from_numpy(coord).cuda(), torch.from_numpy(nlist).cuda(), torch.from_numpy(w.atype).cuda()
    ei = dpc.env_info(*env)
    dD = W.normal(46, (w.nloc, w.M1, w.M2))
    s, Rt, nvalid = dpc.dp_env_mat_df64(cg, ng, w.sel, ei)
    T = dpc.dp_tabulate_fusion_fwd_moments_df64(model.table, model.info, s, Rt, nvalid, at, w.sel)
    dT = dpc.dp_descriptor_contract_grad_df64(T, torch.from_numpy(dD).cuda())
    ds, dRt = dpc.dp_tabulate_fusion_grad_moments_df64(model.table, model.info, s, Rt, nvalid, at, w.sel, dT)
    F, Wv = dpc.dp_force_virial_df64(cg, ng, ei, ds, dRt)
    torch.cuda.synchronize()
    o = oracle.default()
    info, tabs = oracle_tables(w, F64)
    so, Rto = o.env_mat(coord, nlist, *env)
    To = o.fwd(tabs, info, so, Rto, w.nvalid, w.atype, w.sel)
    dso, dRo = o.grad(tabs, info, so, Rto, w.nvalid, w.atype, w.sel, o.descriptor_grad(To, dD))
    Fo, Wo = o.force_virial(coord, nlist, env[0], env[1], dso, dRo, env[2], env[3])
    assert rel(F.cpu().numpy(), Fo) <= TOL[F64] and rel(Wv.cpu().numpy(), Wo) <= TOL[F64]
    folded = np.zeros((w.nloc, 3))
    np.add.at(folded, owner, F.cpu().numpy())
    assert np.abs(folded.sum(axis=0)).max() <= 1e-9 * np.abs(folded).max()


def test_df64_env_edges():
    """A neighbour exactly at rc gives s = 0 and no force; u = 1/2 gives w = 1/2 exactly; padding rows."""
    dpc = lib()
    for kind in (0, 1):
        ei = dpc.env_info(1.0, 3.0, kind=kind)
        coord = torch.tensor([[0.0, 0.0, 0.0], [3.0, 0.0, 0.0], [3.0, 2.0, 0.0]], dtype=F64, device="cuda")
        nl = torch.tensor([[-1, -1, -1, -1], [0, 2, -1, -1]], dtype=torch.int32, device="cuda")
        s, Rt, nv = dpc.dp_env_mat_df64(coord, nl, [4], ei)
        torch.cuda.synchronize()
        assert nv.cpu().tolist() == [[0], [2]]
        assert not s[0].abs().max().item() and s[1, 0].item() == 0.0
        assert abs(s[1, 1].item() - 0.25) <= 1e-15
        F, Wv = dpc.dp_force_virial_df64(coord, nl, ei, torch.ones((2, 4), dtype=F64, device="cuda"),
                                         torch.ones((2, 4, 4), dtype=F64, device="cuda"))
        torch.cuda.synchronize()
        Fo, Wo = oracle.default().force_virial(coord.cpu().numpy(), nl.cpu().numpy(), 1.0, 3.0, np.ones((2, 4)),
                                               np.ones((2, 4, 4)), kind)
        assert rel(F.cpu().numpy(), Fo) <= TOL[F64] and rel(Wv.cpu().numpy(), Wo) <= TOL[F64]
