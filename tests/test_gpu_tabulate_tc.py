"""The f64 tabulated forward and backward with the per-interval contraction on the tensor cores
(dp_tabulate_fusion_{fwd,grad}_tc_f64: interval moments times the scaled table, exact digit-split
GEMMs) against the oracle (Sec. II: T_i = R~_i^T G_i / N_c and its backward), against the FP64-pipe
moment path, and on the edge cases of its own bookkeeping: unsorted rows (a key met twice), several
centre types in any order, chunks of atoms, empty counts, clamped and NaN inputs (GPU).  Tolerance as
for every f64 output: 1e-11 max-norm relative; against the FP64-pipe path, 1e-12."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from gpu_common import TOL, assert_parity, lib, need_gpu, product_model, rel, run_oracle, to_dev, workload

pytestmark = pytest.mark.gpu
F64 = torch.float64
CLOSE = 1e-12  # against the FP64-pipe moment path (same sums, other rounding order)


@pytest.fixture(autouse=True)
def _gpu():
    need_gpu()


def _tc(w, model=None, x=None, nvalid="w", atype="w", work=None, out=None, grad_out=None, reuse=False, plan=None):
    """Forward (writing D as well) then backward on the tensor-core path; reuse: the backward takes the
    forward's interval runs from the shared work buffer (the benchmark's configuration); plan: a TcPlan,
    else the table is planned per call."""
    dpc = lib()
    model = model or product_model(w, F64)
    x = x or to_dev(w, F64)
    nv = x["nvalid"] if isinstance(nvalid, str) else nvalid
    at = x["atype"] if isinstance(atype, str) else atype
    tab = plan if plan is not None else model.table
    if reuse and work is None:
        need = dpc.dp_tabulate_tc_work_bytes(model.info, w.nloc, w.nnei, w.ntypes, w.M1)
        work = torch.empty((need,), dtype=torch.uint8, device="cuda")
    T, D = dpc.dp_tabulate_fusion_fwd_tc_f64(tab, model.info, x["s"], x["Rt"], nv, at, w.sel, out=out, work=work,
                                             M2=w.M2)
    ds, dRt = dpc.dp_tabulate_fusion_grad_tc_f64(tab, model.info, x["s"], x["Rt"], nv, at, w.sel, x["dT"],
                                                 out=grad_out, work=work,
                                                 flags=dpc.DP_TC_REUSE_RUNS if reuse else 0)
    Dc = dpc.dp_descriptor_contract(T, w.M2)  # the same T contracted by the separate call
    torch.cuda.synchronize()
    assert torch.equal(D.view(torch.int64), Dc.view(torch.int64)), "the forward's D differs from dp_descriptor_contract"
    return dict(T=T.cpu().numpy(), D=D.cpu().numpy(), ds=ds.cpu().numpy(), dRt=dRt.cpu().numpy())


def _pipe(w, model, x):
    dpc = lib()
    args = (model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    T = dpc.dp_tabulate_fusion_fwd_moments(*args)
    ds, dRt = dpc.dp_tabulate_fusion_grad_moments(*args, x["dT"])
    torch.cuda.synchronize()
    return dict(T=T.cpu().numpy(), ds=ds.cpu().numpy(), dRt=dRt.cpu().numpy())


CASES = [
    ("tiny", {}, None), ("water", dict(nmol=256), None), ("cu85", dict(cells=(6, 6, 6)), None),
    ("cugeo", dict(cells=(6, 6, 6)), None), ("alcumg", dict(pad=0.1, cells=(6, 6, 6)), None),
    ("alcumg", dict(pad=0.6, cells=(6, 6, 6)), None), ("cu85", {}, None), ("water", {}, 512),
    ("cugeo", {}, 512), ("alcumg", dict(pad=0.1), 384), ("alcumg", dict(pad=0.3), 384),
    ("alcumg", dict(pad=0.6), 384),
]
CHUNK = 16416  # atoms per chunk of the tensor-core calls (their work buffer holds one chunk)


@pytest.mark.parametrize("name,kw,nsample", CASES, ids=[f"{c[0]}-{c[1]}" for c in CASES])
def test_tc_against_oracle_and_fp64_path(name, kw, nsample):
    """T, D (written by the forward), ds and dR~ in the benchmark's configuration (a plan made once, the
    backward reusing the forward's interval runs) against the oracle (sampled atoms at the largest sizes)
    and against the FP64-pipe moment kernels on every atom; bit-identical to a backward that finds the runs
    itself, and D to dp_descriptor_contract of the same T."""
    w = workload(name, **kw)
    model = product_model(w, F64)
    x = to_dev(w, F64)
    plan = lib().dp_tabulate_tc_plan_f64(model.table, model.info, w.nnei)
    got = _tc(w, model, x, reuse=True, plan=plan)
    fresh = _tc(w, model, x)  # the backward finding the runs itself, the table planned per call
    for k in got:
        assert np.array_equal(got[k], fresh[k]), k
    atoms = None
    if nsample:
        atoms = np.sort(np.random.default_rng(5).choice(w.nloc, nsample, replace=False))
        atoms[0], atoms[-1] = 0, w.nloc - 1
    ref = run_oracle(w, F64, atoms=atoms)
    assert_parity(got, ref, F64, atoms=atoms, keys=("T", "D", "ds", "dRt"))
    pipe = _pipe(w, model, x)
    for k in ("T", "ds", "dRt"):
        assert rel(got[k], pipe[k]) <= CLOSE, (k, rel(got[k], pipe[k]))


@pytest.mark.parametrize("M1,widths", [(1, (1, 1)), (37, (1, 5, 37)), (64, (1, 16, 32, 64)), (200, (1, 50, 100, 200)),
                                       (256, (1, 64, 128, 256))])
def test_tc_channel_counts_clamped_and_nan(M1, widths):
    """One to two 128-channel tiles of the forward GEMM, long runs, a row past the coarse segment, one
    below the table and a NaN: the NaN atom's T is NaN and its other rows' gradients are not."""
    w = W.tiny(seed=95 + M1, nloc=11, nreal=27, sel=30, widths=widths, M2=1, rmin=2.6, rmax=3.0)
    s = w.s.copy()
    s[0, 0], s[1, 2], s[2, 1] = w.s_max * 7.0, w.s_min - 1.0, np.nan
    w2 = W.Workload(**{**w.__dict__, "s": s})
    got = _tc(w2, atype=None)
    ref = run_oracle(w2, F64)
    assert np.isnan(got["T"][2]).all() and not np.isnan(np.delete(got["T"], 2, axis=0)).any()
    assert np.isnan(got["ds"][2, 1]) and np.isnan(got["dRt"][2, 1]).all()
    info = oracle.default().table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    for i, j in ((0, 0), (1, 2)):  # clamped rows (past the coarse segment, below the table): no derivative
        if (s[i, j] >= info.upper_ext or s[i, j] < info.lower) and j < w.nvalid[i].sum():
            assert got["ds"][i, j] == 0.0
    keep = np.arange(w2.nloc) != 2
    assert rel(got["T"][keep], ref["T"][keep]) <= TOL[F64]
    for k in ("ds", "dRt"):
        g, r = got[k].copy(), ref[k].copy()
        nan = np.isnan(r)
        assert np.array_equal(np.isnan(g), nan)
        g[nan] = r[nan] = 0.0
        assert rel(g, r) <= TOL[F64], (k, rel(g, r))


def test_tc_rows_at_nodes_and_range_boundaries():
    """s on every node of the grid, one ulp and 1e-9 either side of it, and on the three range boundaries
    (lower, the fine/coarse junction upper, upper_ext) and just either side of them, in random order: the
    per-row kernels take the interval from an f32 view of s, which may pick either interval at a node, and
    the f64 search near the range boundaries; T, ds and dR~ match the oracle, with the backward reusing the
    forward's runs."""
    w = W.tiny(seed=61, nloc=24, nreal=30, sel=32, widths=(1, 8, 16, 32), M2=4)
    info = oracle.default().table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    nodes = [info.lower + l * info.stride0 for l in range(info.n0)]
    nodes += [info.upper + k * info.stride1 for k in range(info.n1 + 1)]
    vals = []
    for x in nodes + [info.lower, info.upper, info.upper_ext]:
        vals += [x, np.nextafter(x, -np.inf), np.nextafter(x, np.inf), x - 1e-9, x + 1e-9]
    rng = np.random.default_rng(3)
    s = w.s.copy()
    nv = w.nvalid.sum(axis=1)
    for i in range(w.nloc):
        s[i, :nv[i]] = rng.choice(np.array(vals), nv[i])
    w2 = W.Workload(**{**w.__dict__, "s": s})
    assert_parity(_tc(w2, atype=None, reuse=True), run_oracle(w2, F64), F64, keys=("T", "ds", "dRt"))


def test_tc_unsorted_rows_many_types_unsorted_centres():
    """ntypes = 8, centre types in random order (several GEMMs share tiles), rows of each segment in
    random order (an interval's rows in several runs add into one slot), some segments empty."""
    rng = np.random.default_rng(12)
    nt = 8
    sel = np.array([5, 0, 7, 3, 9, 1, 4, 6], np.int32)
    nloc = 53
    base = W.tiny(seed=43, nloc=nloc, nreal=0, sel=int(sel.sum()), widths=(1, 4, 8, 16), M2=4)
    s = np.zeros((nloc, sel.sum()))
    Rt = np.zeros((nloc, sel.sum(), 4))
    nvalid = np.zeros((nloc, nt), np.int32)
    off = np.concatenate([[0], np.cumsum(sel)])
    for i in range(nloc):
        for b in range(nt):
            nv = int(rng.integers(0, sel[b] + 1))
            nvalid[i, b] = nv
            sv = rng.uniform(0.01, 1.0, nv)  # not sorted
            s[i, off[b]:off[b] + nv] = sv
            d = rng.normal(size=(nv, 3))
            d /= np.linalg.norm(d, axis=1, keepdims=True)
            Rt[i, off[b]:off[b] + nv, 0] = sv
            Rt[i, off[b]:off[b] + nv, 1:] = sv[:, None] * d
    w = W.Workload(name="types8u", seed=43, ntypes=nt, sel=sel, widths=[1, 4, 8, 16], M2=4, s=s, Rt=Rt,
                   nvalid=nvalid, atype=rng.integers(0, nt, nloc).astype(np.int32),
                   params=W.net_params(78, [1, 4, 8, 16], nt * nt), dT=base.dT, s_min=float(s[s > 0].min()),
                   s_max=float(s.max()))
    ref = run_oracle(w, F64)
    assert_parity(_tc(w), ref, F64, keys=("T", "ds", "dRt"))
    assert_parity(_tc(w, reuse=True), ref, F64, keys=("T", "ds", "dRt"))


def test_tc_empty_counts_and_overwrite():
    """nloc = 0; all counts 0 (T = 0 and zero gradients over stale outputs); NULL counts = all rows valid;
    NaN-prefilled outputs fully overwritten."""
    dpc = lib()
    w = W.water(seed=31, nmol=48, widths=(1, 8, 16, 32), M2=8, sel=(24, 48), rc=5.0)
    model = product_model(w, F64)
    x = to_dev(w, F64)
    e = lambda *shape: torch.empty(shape, dtype=F64, device="cuda")  # noqa: E731
    T0 = dpc.dp_tabulate_fusion_fwd_tc_f64(model.table, model.info, e(0, w.nnei), e(0, w.nnei, 4), None, None, w.sel)
    assert T0.shape == (0, 4, w.M1)
    full = lambda v, *sh: torch.full(sh, v, dtype=F64, device="cuda")  # noqa: E731
    zero = torch.zeros_like(x["nvalid"])
    g = _tc(w, model, x, nvalid=zero, out=full(7.0, w.nloc, 4, w.M1),
            grad_out=(full(7.0, w.nloc, w.nnei), full(-3.0, w.nloc, w.nnei, 4)))
    assert not g["T"].any() and not g["ds"].any() and not g["dRt"].any()
    allv = torch.tensor(np.broadcast_to(w.sel, w.nvalid.shape).copy(), dtype=torch.int32, device="cuda")
    a = _tc(w, model, x, nvalid=allv)
    b = _tc(w, model, x, nvalid=None, out=full(np.nan, w.nloc, 4, w.M1),
            grad_out=(full(np.nan, w.nloc, w.nnei), full(np.nan, w.nloc, w.nnei, 4)))
    for k in ("T", "ds", "dRt"):
        assert np.array_equal(a[k], b[k]) and not np.isnan(b[k]).any()


def test_tc_chunks_of_atoms():
    """More atoms than one chunk (16,416), with a ragged last chunk, against the FP64-pipe path, and the
    oracle on atoms at the chunk edges; the backward reusing the forward's runs of every chunk gives the
    same bits as one that finds them itself."""
    w = workload("water", nmol=6000)  # 18,000 atoms
    model = product_model(w, F64)
    x = to_dev(w, F64)
    got = _tc(w, model, x, reuse=True)
    fresh = _tc(w, model, x)
    for k in got:
        assert np.array_equal(got[k], fresh[k]), k
    pipe = _pipe(w, model, x)
    for k in ("T", "ds", "dRt"):
        assert rel(got[k], pipe[k]) <= CLOSE, k
    atoms = np.r_[0:4, CHUNK - 4:CHUNK + 4, w.nloc - 4:w.nloc]
    assert_parity(got, run_oracle(w, F64, atoms=atoms), F64, atoms=atoms, keys=("T", "ds", "dRt"))


def test_tc_work_buffer_rules_and_reuse():
    """The size query (one size for both directions), a short or misaligned buffer refused on the host,
    a plan made for another geometry refused, and repeated calls on one dirty buffer giving bit-identical
    results, with and without the backward reusing the forward's runs."""
    dpc = lib()
    w = workload("water", nmol=256)
    model = product_model(w, F64)
    x = to_dev(w, F64)
    need = dpc.dp_tabulate_tc_work_bytes(model.info, w.nloc, w.nnei, w.ntypes, w.M1)
    assert need > 0 and need % 256 == 0
    work = torch.empty((need + 256,), dtype=torch.uint8, device="cuda")
    a = _tc(w, model, x, work=work[:need])
    for reuse in (False, True):
        work.fill_(0xff)
        b = _tc(w, model, x, work=work[:need], reuse=reuse)
        for k in a:
            assert np.array_equal(a[k], b[k]), (k, reuse)
    other = dpc.dp_tabulate_tc_plan_f64(model.table, model.info, w.nnei + 1)
    with pytest.raises(dpc.DPError):
        dpc.dp_tabulate_fusion_fwd_tc_f64(other, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel,
                                          work=work[:need])
    args = (model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    with pytest.raises(ValueError):
        dpc.dp_tabulate_fusion_fwd_tc_f64(*args, work=work[:need - 1])
    with pytest.raises(dpc.DPError):
        dpc.dp_tabulate_fusion_fwd_tc_f64(*args, work=work[16:need + 16])
    with pytest.raises(ValueError):
        dpc.dp_tabulate_tc_work_bytes(model.info, w.nloc, 0, w.ntypes, w.M1)
    assert dpc.dp_tc_wait_timeouts() == 0  # no bounded wait of the GEMM kernels gave up


def test_tc_water_large_chunk_edges():
    """The default f64 path at its largest size: 1,048,576 atoms in 64 chunks, in the benchmark's launch
    configuration (one plan, one work buffer, the backward reusing the forward's interval runs).  The
    oracle on 256 atoms gathered on the device: the first and last atom of 24 chunks spread over the run (edges from the 1st chunk to the 64th, byte offsets into R~ and dR~ past
    2^32) and random atoms; the FP64-pipe moment path on every atom, compared on the device; and
    the identity <dR~, R~> = <dT, T> over every atom, which holds at any size."""
    dpc = lib()
    w = workload("water_large")
    nchunks = -(-w.nloc // CHUNK)
    assert nchunks >= 64
    model = product_model(w, F64)
    x = to_dev(w, F64)
    args = (model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    plan = dpc.dp_tabulate_tc_plan_f64(model.table, model.info, w.nnei)
    pargs = (plan,) + args[1:]
    work = torch.empty((dpc.dp_tabulate_tc_work_bytes(model.info, w.nloc, w.nnei, w.ntypes, w.M1),),
                       dtype=torch.uint8, device="cuda")
    T = dpc.dp_tabulate_fusion_fwd_tc_f64(*pargs, work=work)
    ds, dRt = dpc.dp_tabulate_fusion_grad_tc_f64(*pargs, x["dT"], work=work, flags=dpc.DP_TC_REUSE_RUNS)
    torch.cuda.synchronize()
    edges = []
    for c in np.unique(np.r_[1, 2, 3, np.linspace(4, nchunks - 1, 21).astype(int)]):
        edges += [c * CHUNK - 1, min(c * CHUNK, w.nloc - 1)]
    rest = np.random.default_rng(17).choice(w.nloc, 256 - len(edges) - 2, replace=False)
    atoms = np.unique(np.r_[0, w.nloc - 1, edges, rest])
    idx = torch.from_numpy(atoms).cuda()
    got = {k: v.index_select(0, idx).cpu().numpy() for k, v in dict(T=T, ds=ds, dRt=dRt).items()}
    assert_parity(got, run_oracle(w, F64, atoms=atoms), F64, keys=("T", "ds", "dRt"))
    lhs = float((dRt * x["Rt"]).sum())
    rhs = float((x["dT"] * T).sum())
    assert abs(lhs - rhs) <= TOL[F64] * 10 * max(1.0, abs(rhs)), (lhs, rhs)
    Tp = dpc.dp_tabulate_fusion_fwd_moments(*args)
    d = float((Tp - T).abs().max() / Tp.abs().max())
    assert d <= CLOSE, ("T", d)
    del Tp
    dsp, dRtp = dpc.dp_tabulate_fusion_grad_moments(*args, x["dT"])
    for k, a, b in (("ds", ds, dsp), ("dRt", dRt, dRtp)):
        d = float((a - b).abs().max() / b.abs().max())
        assert d <= CLOSE, (k, d)
    assert dpc.dp_tc_wait_timeouts() == 0
    del T, ds, dRt, dsp, dRtp, x, model, work, plan
    torch.cuda.empty_cache()


@pytest.mark.parametrize("M2", [1, 7, 32])
def test_tc_descriptor_widths(M2):
    """D written by the tensor-core forward at M2 = 1, an odd width and M2 = M1: bit for bit
    dp_descriptor_contract of the same T, and the oracle's D; M2 = 0 or M2 > M1 refused."""
    dpc = lib()
    w = W.water(seed=33, nmol=64, widths=(1, 8, 16, 32), M2=4, sel=(24, 48), rc=5.0)
    model = product_model(w, F64)
    x = to_dev(w, F64)
    args = (model.table, model.info, x["s"], x["Rt"], x["nvalid"], x["atype"], w.sel)
    T, D = dpc.dp_tabulate_fusion_fwd_tc_f64(*args, M2=M2)
    Dc = dpc.dp_descriptor_contract(T, M2)
    torch.cuda.synchronize()
    assert D.shape == (w.nloc, w.M1, M2)
    assert torch.equal(D.view(torch.int64), Dc.view(torch.int64))
    Do = oracle.default().descriptor(T.cpu().numpy(), M2)
    assert rel(D.cpu().numpy(), Do) <= 1e-14
    for bad in (0, w.M1 + 1):
        with pytest.raises(ValueError):
            dpc.dp_tabulate_fusion_fwd_tc_f64(*args, M2=bad)
