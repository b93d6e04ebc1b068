"""CUDA path vs the oracle, element by element, on the same seeded inputs (GPU).

Tolerance (max-norm relative per output array): 1e-11 in f64, 2e-5 in f32.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import (TOL, assert_parity, lib, need_gpu, oracle_tables, product_model, rel, run_oracle,
                        run_product, to_dev, workload)

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


# ------------------------------------------------------------------ compression

def test_table_info_matches_oracle():
    dpc = lib()
    o = oracle.default()
    for smin, smax in ((0.0, 1.05), (0.003, 0.52), (-0.237, 0.42), (1e-9, 1.1)):
        a = dpc.dp_table_info_make(smin, smax, 0.01, 0.1, 5.0)
        b = o.table_info(smin, smax, 0.01, 0.1, 5.0)
        assert (a.lower, a.upper, a.upper_ext, a.stride0, a.stride1) == b.as_tuple()
        assert dpc.dp_table_info_sizes(a) == (b.n0, b.n1)


@pytest.mark.parametrize("name", ["tiny", "water_s"])
def test_nodes_and_table(name):
    """Net nodes vs the oracle's (long double); the table build vs the oracle's on the SAME nodes, compared on
    evaluated g, g', g'' at both ends and inside each interval (raw coefficients are cancellation-heavy)."""
    dpc = lib()
    o = oracle.default()
    w = workload("tiny") if name == "tiny" else workload("water", nmol=64, sel=(40, 80))
    info_o = o.table_info(w.s_min, w.s_max)
    info = dpc.dp_table_info_make(w.s_min, w.s_max)
    params = torch.from_numpy(w.params).cuda()
    y, dy, d2y = dpc.dp_embedding_net_nodes(params, w.widths, info)
    tab64 = dpc.dp_table_build(y, dy, d2y, info, torch.float64)
    tab32 = dpc.dp_table_build(y, dy, d2y, info, torch.float32)
    torch.cuda.synchronize()
    for p in range(w.npair):
        ry, rdy, rd2y = o.nodes(w.params[p], w.widths, info_o)
        gy, gdy, gd2y = (a[p].cpu().numpy() for a in (y, dy, d2y))
        assert rel(gy, ry) < 1e-14 and rel(gdy, rdy) < 1e-13 and rel(gd2y, rd2y) < 1e-12
        same = o.table_build(gy, gdy, gd2y, info_o)     # oracle build on the GPU's nodes
        full = o.table_build(ry, rdy, rd2y, info_o)     # oracle nodes and build
        g64 = dpc.table_rows(tab64)[p].cpu().numpy()
        g32 = dpc.table_rows(tab32)[p].cpu().numpy().astype(np.float64)
        for l in list(range(0, info_o.nint, 7)) + [info_o.n0 - 1, info_o.n0, info_o.nint - 1]:
            Dt = info_o.stride0 if l < info_o.n0 else info_o.stride1
            for t in (0.0, 0.37 * Dt, Dt):
                for order in range(3):
                    r = o.poly_eval(same, l, t, order)
                    scale = np.abs(r).max() + 1e-300
                    # same nodes: only the build's own rounding remains
                    assert np.abs(o.poly_eval(g64, l, t, order) - r).max() / scale < (1e-14, 1e-13, 1e-12)[order]
                    # different nodes: a node change of eps*|y| moves g^(k) by ~eps*|y|/Dt^k
                    rf = o.poly_eval(full, l, t, order)
                    lim = 1e-14 * (1.0, 10.0 / Dt, 100.0 / Dt ** 2)[order]
                    assert np.abs(o.poly_eval(g64, l, t, order) - rf).max() / (np.abs(rf).max() + 1e-300) < lim
                    if order == 0:
                        assert np.abs(o.poly_eval(g32, l, t, 0) - r).max() / scale < 1e-6


# ------------------------------------------------------------------ path parity

CASES = [
    ("tiny", {}, torch.float64),
    ("tiny", {}, torch.float32),
    ("water", dict(nmol=256), torch.float64),
    ("water", dict(nmol=256), torch.float32),
    ("cu85", dict(cells=(6, 6, 6)), torch.float64),
    ("cugeo", dict(cells=(6, 6, 6)), torch.float64),
    ("alcumg", dict(pad=0.1, cells=(6, 6, 6)), torch.float64),
    ("alcumg", dict(pad=0.6, cells=(6, 6, 6)), torch.float64),
    ("alcumg", dict(pad=0.3, cells=(6, 6, 6)), torch.float32),
]


@pytest.mark.parametrize("name,kw,dtype", CASES, ids=[f"{c[0]}-{c[1]}-{str(c[2])[6:]}" for c in CASES])
def test_path_parity(name, kw, dtype):
    w = workload(name, **kw)
    got = run_product(w, dtype)
    ref = run_oracle(w, dtype)
    assert_parity(got, ref, dtype)


@pytest.mark.parametrize("M1,widths", [(1, (1, 1)), (7, (1, 7)), (37, (1, 5, 37)), (64, (1, 16, 32, 64)),
                                       (128, (1, 32, 64, 128)), (200, (1, 50, 100, 200)),
                                       (256, (1, 64, 128, 256))])
@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_channel_counts(M1, widths, dtype):
    """Every forward kernel shape (CL, R) and ragged channel tails."""
    w = W.tiny(seed=20 + M1, nloc=13, nreal=21, sel=29, widths=widths, M2=min(4, M1))
    assert_parity(run_product(w, dtype), run_oracle(w, dtype), dtype)


def test_many_types_unsorted_centres():
    """ntypes = 8 (the limit), centre types in random order, some segments empty or full."""
    rng = np.random.default_rng(2)
    nt = 8
    sel = np.array([5, 0, 7, 3, 9, 1, 4, 6], np.int32)
    base = W.tiny(seed=41, nloc=37, nreal=0, sel=int(sel.sum()), widths=(1, 4, 8, 16), M2=4)
    s = np.zeros((37, sel.sum()))
    Rt = np.zeros((37, sel.sum(), 4))
    nvalid = np.zeros((37, nt), np.int32)
    off = np.concatenate([[0], np.cumsum(sel)])
    for i in range(37):
        for b in range(nt):
            nv = int(rng.integers(0, sel[b] + 1))
            nvalid[i, b] = nv
            sv = np.sort(rng.uniform(0.01, 1.0, nv))[::-1]
            s[i, off[b]:off[b] + nv] = sv
            d = rng.normal(size=(nv, 3))
            d /= np.linalg.norm(d, axis=1, keepdims=True)
            Rt[i, off[b]:off[b] + nv, 0] = sv
            Rt[i, off[b]:off[b] + nv, 1:] = sv[:, None] * d
    w = W.Workload(name="types8", seed=41, ntypes=nt, sel=sel, widths=[1, 4, 8, 16], M2=4, s=s, Rt=Rt,
                   nvalid=nvalid, atype=rng.integers(0, nt, 37).astype(np.int32),
                   params=W.net_params(77, [1, 4, 8, 16], nt * nt), dT=base.dT, s_min=float(s[s > 0].min()),
                   s_max=float(s.max()))
    for dtype in (torch.float64, torch.float32):
        assert_parity(run_product(w, dtype), run_oracle(w, dtype), dtype)


# ------------------------------------------------------------------- edge cases

def _edge_workload():
    return W.water(seed=31, nmol=48, widths=(1, 8, 16, 32), M2=8, sel=(24, 48), rc=5.0)


def test_empty_and_degenerate_counts():
    dpc = lib()
    w = _edge_workload()
    for dtype in (torch.float64, torch.float32):
        model = product_model(w, dtype)
        x = to_dev(w, dtype)
        # nloc = 0: nothing to do, DP_OK
        e = lambda *shape: torch.empty(shape, dtype=dtype, device="cuda")  # noqa: E731
        T0 = dpc.dp_tabulate_fusion_fwd(model.table, model.info, e(0, w.nnei), e(0, w.nnei, 4),
                                        torch.empty((0, 2), dtype=torch.int32, device="cuda"), None, w.sel)
        assert T0.shape == (0, 4, w.M1)
        # all counts 0: T = 0, all grads 0
        zero = torch.zeros_like(x["nvalid"])
        T = torch.full((w.nloc, 4, w.M1), 7.0, dtype=dtype, device="cuda")
        dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], zero, x["atype"], w.sel, out=T)
        ds, dRt = dpc.dp_tabulate_fusion_grad(model.table, model.info, x["s"], x["Rt"], zero, x["atype"], w.sel,
                                              x["dT"])
        assert torch.count_nonzero(T) == 0 and torch.count_nonzero(ds) == 0 and torch.count_nonzero(dRt) == 0
        # counts = sel (padding processed) equals the skipping run; NULL counts mean all rows valid
        full = torch.tensor(np.broadcast_to(w.sel, w.nvalid.shape).copy(), dtype=torch.int32, device="cuda")
        Ta = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
        Tb = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], full, x["atype"], w.sel)
        Tc = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], None, x["atype"], w.sel)
        assert rel(Tb.cpu(), Ta.cpu()) < TOL[dtype] and torch.equal(Tb, Tc)
        # counts above sel are clamped to sel
        big = (full + 1000).contiguous()
        Td = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], big, x["atype"], w.sel)
        assert torch.equal(Td, Tb)


def test_clamped_coarse_and_nan_inputs():
    """s in the coarse segment, above upper_ext, below lower, and NaN, against the oracle."""
    w = _edge_workload()
    s, Rt = w.s.copy(), w.Rt.copy()
    rng = np.random.default_rng(9)
    info_hi = None
    rows = []
    for i in range(w.nloc):
        for b, off in ((0, 0), (1, w.sel[0])):
            for j in range(w.nvalid[i, b]):
                rows.append((i, off + j))
    rows = np.array(rows)
    pick = rows[rng.choice(len(rows), 60, replace=False)]
    o = oracle.default()
    info = o.table_info(w.s_min, w.s_max)
    vals = [info.upper + 0.37, info.upper + 2.0, info.upper_ext - 1e-9, info.upper_ext, info.upper_ext + 3.0,
            info.lower - 0.25, info.upper - 1e-12, info.upper]
    for q, (i, r) in enumerate(pick[:-1]):
        s[i, r] = vals[q % len(vals)]
    nan_atom, nan_row = pick[-1]
    s[nan_atom, nan_row] = np.nan
    w2 = W.Workload(**{**w.__dict__, "s": s, "Rt": Rt})
    for dtype in (torch.float64, torch.float32):
        got = run_product(w2, dtype)
        ref = run_oracle(w2, dtype)
        assert np.all(np.isnan(got["T"][nan_atom])) and np.all(np.isnan(ref["T"][nan_atom]))
        assert np.isnan(got["ds"][nan_atom, nan_row]) and np.all(np.isnan(got["dRt"][nan_atom, nan_row]))
        keep = np.ones(w.nloc, bool)
        keep[nan_atom] = False
        for k in ("T", "D", "ds", "dRt"):
            g, r_ = got[k][keep], ref[k][keep]
            assert rel(g, r_) <= TOL[dtype], (k, rel(g, r_))
        # the NaN atom's other rows are finite and match
        other = np.ones(w.nnei, bool)
        other[nan_row] = False
        assert rel(got["ds"][nan_atom, other], ref["ds"][nan_atom, other]) <= TOL[dtype]
        # clamped rows: ds exactly 0
        for (i, r), v in zip(pick[:-1], [vals[q % len(vals)] for q in range(len(pick) - 1)]):
            if v >= info.upper_ext or v < info.lower:
                assert got["ds"][i, r] == 0.0


def test_ragged_atom_counts():
    """nloc not a multiple of the block's atoms, nnei not a multiple of the grad block."""
    for nloc in (1, 2, 3, 5, 130):
        w = W.tiny(seed=60 + nloc, nloc=nloc, nreal=17, sel=131, widths=(1, 4, 8, 16), M2=4)
        for dtype in (torch.float64, torch.float32):
            assert_parity(run_product(w, dtype), run_oracle(w, dtype), dtype)


def test_output_fully_overwritten():
    """Outputs prefilled with NaN: every element is written (padding rows included)."""
    dpc = lib()
    w = _edge_workload()
    for dtype in (torch.float64, torch.float32):
        model = product_model(w, dtype)
        x = to_dev(w, dtype)
        nan = lambda *sh: torch.full(sh, float("nan"), dtype=dtype, device="cuda")  # noqa: E731
        T = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel,
                                       out=nan(w.nloc, 4, w.M1))
        ds, dRt = dpc.dp_tabulate_fusion_grad(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"],
                                              w.sel, x["dT"], out=(nan(w.nloc, w.nnei), nan(w.nloc, w.nnei, 4)))
        D = dpc.dp_descriptor_contract(T, w.M2, out=nan(w.nloc, w.M1, w.M2))
        for t in (T, ds, dRt, D):
            assert not torch.isnan(t).any()


# ---------------------------------------------------------- paper-sized inputs

@pytest.mark.parametrize("name,kw,dtype,nsample", [
    ("cu85", {}, torch.float64, None),
    ("water", {}, torch.float64, None),
    ("water", {}, torch.float32, None),
    ("cugeo", {}, torch.float64, 512),
    ("alcumg", dict(pad=0.1), torch.float64, 384),
    ("alcumg", dict(pad=0.6), torch.float64, 384),
])
def test_paper_sized(name, kw, dtype, nsample):
    """Full-size workloads in the benchmark's launch configuration; sampled atoms where the oracle is slow."""
    w = workload(name, **kw)
    got = run_product(w, dtype)
    atoms = None
    if nsample is not None:
        rng = np.random.default_rng(1)
        atoms = np.sort(rng.choice(w.nloc, nsample, replace=False))
        atoms[0], atoms[-1] = 0, w.nloc - 1
    ref = run_oracle(w, dtype, atoms=atoms)
    assert_parity(got, ref, dtype, atoms=atoms)


@pytest.mark.parametrize("pad", [0.2, 0.3, 0.4, 0.5])
def test_alcumg_padding_sweep(pad):
    """The Al-Cu-Mg-like padding sweep (10-60 % empty rows), small cells, every atom."""
    w = workload("alcumg", pad=pad, cells=(6, 6, 6))
    assert_parity(run_product(w, torch.float64), run_oracle(w, torch.float64), torch.float64)


@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_water_large_sampled(dtype):
    """1,048,576 atoms in the benchmark's launch configuration; 256 sampled atoms (first and last
    included) gathered on the device and compared with the oracle; plus the identity
    <dR~, R~> = <dT, T> over ALL atoms, which holds at any size."""
    dpc = lib()
    w = workload("water_large")
    model = product_model(w, dtype)
    x = to_dev(w, dtype)
    T = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    D = dpc.dp_descriptor_contract(T, w.M2)
    ds, dRt = dpc.dp_tabulate_fusion_grad(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel,
                                          x["dT"])
    torch.cuda.synchronize()
    rng = np.random.default_rng(7)
    atoms = np.sort(rng.choice(w.nloc, 256, replace=False))
    atoms[0], atoms[-1] = 0, w.nloc - 1
    idx = torch.from_numpy(atoms).cuda()
    got = {k: v.index_select(0, idx).double().cpu().numpy() for k, v in dict(T=T, D=D, ds=ds, dRt=dRt).items()}
    ref = run_oracle(w, dtype, atoms=atoms)
    assert_parity(got, ref, dtype)
    lhs = float((dRt.double() * x["Rt"].double()).sum())
    rhs = float((x["dT"].double() * T.double()).sum())
    assert abs(lhs - rhs) <= TOL[dtype] * 10 * max(1.0, abs(rhs)), (lhs, rhs)
    del T, D, ds, dRt, x, model
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_normalised_environment_matrix(dtype):
    """The paper's normalisation of the 4-vectors (s shifted by its mean and scaled by its std, the
    xyz columns by their joint std): s takes negative values, so the table starts below zero."""
    base = W.water(seed=52, nmol=128, widths=(1, 8, 16, 32), M2=8)
    off = np.concatenate([[0], np.cumsum(base.sel)])
    valid = np.zeros(base.s.shape, bool)
    for b in range(base.ntypes):
        valid[:, off[b]:off[b + 1]] = np.arange(base.sel[b])[None, :] < base.nvalid[:, b:b + 1]
    sv = base.s[valid]
    xyz = base.Rt[..., 1:][valid]
    norm = (float(sv.mean()), float(sv.std()), float(xyz.std()))
    w = W.water(seed=52, nmol=128, widths=(1, 8, 16, 32), M2=8, norm=norm)
    assert w.s_min < 0.0
    got = run_product(w, dtype)
    ref = run_oracle(w, dtype)
    assert_parity(got, ref, dtype)


MOMENT_CASES = [
    ("tiny", {}, torch.float64, None), ("tiny", {}, torch.float32, None),
    ("water", dict(nmol=256), torch.float64, None), ("water", dict(nmol=256), torch.float32, None),
    ("cu85", dict(cells=(6, 6, 6)), torch.float64, None), ("cu85", dict(cells=(6, 6, 6)), torch.float32, None),
    ("alcumg", dict(pad=0.1, cells=(6, 6, 6)), torch.float64, None),
    ("cu85", {}, torch.float64, None), ("alcumg", dict(pad=0.3), torch.float64, 384),
    ("cu85", {}, torch.float32, None), ("water", {}, torch.float32, 512),
]


@pytest.mark.parametrize("name,kw,dtype,nsample", MOMENT_CASES,
                         ids=[f"{c[0]}-{c[1]}-{str(c[2])[6:]}" for c in MOMENT_CASES])
def test_moments_forward(name, kw, dtype, nsample):
    """The interval-moment forward gives the oracle's T (and equals the per-neighbour forward up to rounding)."""
    dpc = lib()
    w = workload(name, **kw)
    model = product_model(w, dtype)
    x = to_dev(w, dtype)
    T = dpc.dp_tabulate_fusion_fwd_moments(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    T0 = dpc.dp_tabulate_fusion_fwd(model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    torch.cuda.synchronize()
    atoms = None
    if nsample:
        rng = np.random.default_rng(3)
        atoms = np.sort(rng.choice(w.nloc, nsample, replace=False))
    ref = run_oracle(w, dtype, atoms=atoms)
    got = T.double().cpu().numpy()
    assert rel(got if atoms is None else got[atoms], ref["T"]) <= TOL[dtype]
    assert rel(got, T0.double().cpu().numpy()) <= TOL[dtype]


@pytest.mark.parametrize("M1,widths", [(1, (1, 1)), (37, (1, 5, 37)), (64, (1, 16, 32, 64)), (200, (1, 50, 100, 200))])
def test_moments_forward_shapes(M1, widths):
    """Long runs (neighbours bunched in s) through every channel-round shape of the moment path."""
    dpc = lib()
    w = W.tiny(seed=90 + M1, nloc=11, nreal=27, sel=30, widths=widths, M2=1, rmin=2.6, rmax=3.0)
    for dtype in (torch.float64, torch.float32):
        model = product_model(w, dtype)
        x = to_dev(w, dtype)
        T = dpc.dp_tabulate_fusion_fwd_moments(model.table, model.info, x["s"], x["Rt"], x["nvalid"], None, w.sel)
        torch.cuda.synchronize()
        assert rel(T.double().cpu().numpy(), run_oracle(w, dtype)["T"]) <= TOL[dtype]


@pytest.mark.parametrize("name,kw,dtype,nsample", MOMENT_CASES,
                         ids=[f"{c[0]}-{c[1]}-{str(c[2])[6:]}" for c in MOMENT_CASES])
def test_moments_grad(name, kw, dtype, nsample):
    """The interval-moment backward gives the oracle's ds and dR~, padding rows zeroed over stale outputs."""
    dpc = lib()
    w = workload(name, **kw)
    model = product_model(w, dtype)
    x = to_dev(w, dtype)
    args = (model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel, x["dT"])
    stale = (torch.full((w.nloc, w.nnei), 7.0, dtype=dtype, device="cuda"),
             torch.full((w.nloc, w.nnei, 4), -3.0, dtype=dtype, device="cuda"))
    ds, dRt = dpc.dp_tabulate_fusion_grad_moments(*args, out=stale)
    ds0, dRt0 = dpc.dp_tabulate_fusion_grad(*args)
    torch.cuda.synchronize()
    atoms = None
    if nsample:
        rng = np.random.default_rng(4)
        atoms = np.sort(rng.choice(w.nloc, nsample, replace=False))
    ref = run_oracle(w, dtype, atoms=atoms)
    got = dict(ds=ds.double().cpu().numpy(), dRt=dRt.double().cpu().numpy())
    assert_parity(got, ref, dtype, atoms=atoms, keys=("ds", "dRt"))
    assert rel(got["ds"], ds0.double().cpu().numpy()) <= TOL[dtype]
    assert rel(got["dRt"], dRt0.double().cpu().numpy()) <= TOL[dtype]


@pytest.mark.parametrize("M1,widths", [(1, (1, 1)), (37, (1, 5, 37)), (64, (1, 16, 32, 64)), (200, (1, 50, 100, 200)),
                                       (256, (1, 64, 128, 256))])
def test_moments_grad_shapes(M1, widths):
    """Long runs and every channel-round shape of the moment backward, with clamped and NaN inputs."""
    dpc = lib()
    w = W.tiny(seed=95 + M1, nloc=11, nreal=27, sel=30, widths=widths, M2=1, rmin=2.6, rmax=3.0)
    s = w.s.copy()
    s[0, 0], s[1, 2], s[2, 1] = w.s_max * 7.0, w.s_min - 1.0, np.nan  # past the coarse segment, below, NaN
    w2 = W.Workload(**{**w.__dict__, "s": s})
    for dtype in (torch.float64, torch.float32):
        model = product_model(w2, dtype)
        x = to_dev(w2, dtype)
        ds, dRt = dpc.dp_tabulate_fusion_grad_moments(model.table, model.info, x["s"], x["Rt"], x["nvalid"], None,
                                                      w2.sel, x["dT"])
        torch.cuda.synchronize()
        ref = run_oracle(w2, dtype)
        got = dict(ds=ds.double().cpu().numpy(), dRt=dRt.double().cpu().numpy())
        nan = np.isnan(ref["ds"])
        assert np.array_equal(np.isnan(got["ds"]), nan)
        got["ds"][nan] = ref["ds"][nan] = 0.0
        nanr = np.isnan(ref["dRt"])
        assert np.array_equal(np.isnan(got["dRt"]), nanr)
        got["dRt"][nanr] = ref["dRt"][nanr] = 0.0
        assert_parity(got, ref, dtype, keys=("ds", "dRt"))


@pytest.mark.parametrize("dtype", [torch.float64, torch.float32])
def test_moments_grad_no_valid_rows(dtype):
    """Atoms without real neighbours: every row is padding and gets zeros over stale outputs, and T is
    zero, in f64 and f32."""
    dpc = lib()
    w = W.tiny(seed=7, nloc=3, nreal=5, sel=80)
    model = product_model(w, dtype)
    x = to_dev(w, dtype)
    stale = (torch.ones((w.nloc, w.nnei), dtype=dtype, device="cuda"),
             torch.ones((w.nloc, w.nnei, 4), dtype=dtype, device="cuda"))
    nv0 = torch.zeros_like(x["nvalid"])
    ds, dRt = dpc.dp_tabulate_fusion_grad_moments(model.table, model.info, x["s"], x["Rt"], nv0, x["atype"], w.sel,
                                                  x["dT"], out=stale)
    T = dpc.dp_tabulate_fusion_fwd_moments(model.table, model.info, x["s"], x["Rt"], nv0, x["atype"], w.sel,
                                           out=torch.ones((w.nloc, 4, w.M1), dtype=dtype, device="cuda"))
    torch.cuda.synchronize()
    assert not ds.abs().max().item() and not dRt.abs().max().item() and not T.abs().max().item()
