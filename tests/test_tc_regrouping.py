"""The arithmetic of the tensor-core tabulation, restated in numpy on the CPU and held against the
oracle (Sec. II: T_i = R~_i^T G_i / N_c and its backward): per interval l of an atom's rows, the
moments W[k][q] = sum_j R~_jk u_j^q with u = t / Delta_l, the scaled coefficients
c'_q = c_q Delta_l^q, T[k][m] = (1/N_c) sum_(l,q) W[k][q] c'_q[m]; backward on the unscaled
coefficients, dW[k][q] = (1/N_c) sum_m dT[k][m] c_q[m], dE/dR~_jk = sum_q dW[k][q] t_j^q and
dE/ds_j = sum_k R~_jk sum_q q dW[k][q] t_j^(q-1) (0 for clamped s).  These are the sums the GPU
GEMMs compute (in exact digit-split form); a dropped power of Delta, the backward on the forward's
scaled coefficients, a wrong factor q or a missing clamp fails here, before any GPU run.  CPU only."""
import numpy as np
import pytest

import oracle
import workloads as W

TOL = 1e-12


def regrouped(o, tabs, info, w, dT, scale_delta=True, q_factor=True, bwd_scaled=False):
    """T, ds, dR~ by interval moments and scaled coefficients, the backward in t on the unscaled
    ones (rows need not be sorted); the switches plant a slip (the forward's coefficients left
    unscaled, the derivative without its factor q, the backward on the scaled coefficients)."""
    nloc, nnei = w.s.shape
    M1 = tabs.shape[-2]
    off = np.concatenate([[0], np.cumsum(w.sel)])
    T = np.zeros((nloc, 4, M1))
    ds = np.zeros((nloc, nnei))
    dR = np.zeros((nloc, nnei, 4))
    for i in range(nloc):
        alpha = int(w.atype[i]) if w.atype is not None else 0
        rows = {}  # key (b, l) -> [(row, u, clamped)]
        for b in range(w.ntypes):
            for j in range(off[b], off[b] + int(w.nvalid[i, b])):
                l, t, clamped = o.locate(info, w.s[i, j])
                delta = info.stride0 if l < info.n0 else info.stride1
                rows.setdefault((b, l), []).append((j, t, t / delta, clamped))
        for (b, l), rr in rows.items():
            delta = info.stride0 if l < info.n0 else info.stride1
            c = tabs[alpha * w.ntypes + b, l]                          # [M1][6]: t^5 .. t^0
            cp = np.stack([c[:, 5 - q] * (delta ** q if scale_delta else 1.0) for q in range(6)])  # c'_q
            ct = np.stack([c[:, 5 - q] for q in range(6)])             # c_q
            Wm = np.zeros((4, 6))
            for j, _, u, _ in rr:
                Wm += np.outer(w.Rt[i, j], u ** np.arange(6))
            T[i] += Wm @ cp / nnei
            dW = dT[i] @ (cp if bwd_scaled else ct).T / nnei           # [4][6]
            for j, t, _, clamped in rr:
                dR[i, j] = dW @ (t ** np.arange(6))
                dq = dW[:, 1:] @ ((np.arange(1, 6) if q_factor else 1.0) * t ** np.arange(5))
                ds[i, j] = 0.0 if clamped else float(w.Rt[i, j] @ dq)
    return T, ds, dR


def _check(w):
    o = oracle.default()
    info = o.table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    tabs = o.tables(w.params, w.widths, info)
    T, ds, dR = regrouped(o, tabs, info, w, w.dT)
    To = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    dso, dRo = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, w.dT)
    for got, ref in ((T, To), (ds, dso), (dR, dRo)):
        err = np.max(np.abs(got - ref)) / np.max(np.abs(ref))
        assert err <= TOL, err


def test_regrouping_matches_oracle_sorted_rows():
    _check(W.tiny(seed=3, nloc=12, nreal=20, sel=24, widths=(1, 4, 8, 16), M2=4))


def test_regrouping_matches_oracle_two_types_unsorted_clamped():
    """Two neighbour types and two centre types, rows shuffled inside their segments (an interval's
    rows in several runs), and rows past the coarse segment and below the table (clamped)."""
    w = W.water(seed=17, nmol=48, widths=(1, 4, 8), M2=4, sel=(24, 48), rc=5.0)
    rng = np.random.default_rng(5)
    s, Rt = w.s.copy(), w.Rt.copy()
    off = np.concatenate([[0], np.cumsum(w.sel)])
    for i in range(w.nloc):
        for b in range(w.ntypes):
            nv = int(w.nvalid[i, b])
            p = off[b] + rng.permutation(nv)
            s[i, off[b]:off[b] + nv], Rt[i, off[b]:off[b] + nv] = s[i, p], Rt[i, p]
    o = oracle.default()
    info = o.table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    s[0, 0] = info.upper_ext + 1.0
    s[1, 1] = info.lower - 0.5
    w2 = W.Workload(**{**w.__dict__, "s": s, "Rt": Rt})
    _check(w2)


@pytest.mark.parametrize("mistake", ["unscaled_coefficients", "no_q_factor", "backward_scaled"])
def test_regrouping_slips_are_caught(mistake):
    """The comparison above notices a plausible slip in the regrouping itself."""
    w = W.tiny(seed=4, nloc=6, nreal=16, sel=16, widths=(1, 4, 8), M2=4)
    o = oracle.default()
    info = o.table_info(w.s_min, w.s_max, w.stride0, w.stride1, w.ext)
    tabs = o.tables(w.params, w.widths, info)
    To = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    dso, _ = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, w.dT)
    kw = {"unscaled_coefficients": {"scale_delta": False}, "no_q_factor": {"q_factor": False},
          "backward_scaled": {"bwd_scaled": True}}[mistake]
    T, ds, _ = regrouped(o, tabs, info, w, w.dT, **kw)
    rel = lambda a, b: np.max(np.abs(a - b)) / np.max(np.abs(b))  # noqa: E731
    assert max(rel(T, To), rel(ds, dso)) > 1e-3


def test_tc_work_and_plan_size_queries():
    """dp_tabulate_tc_work_bytes and dp_tabulate_tc_plan_bytes on the host: one work size for both
    directions, 256-byte multiples; the work grows with the atoms by the chunk's scratch until the
    chunk (16,416 atoms) caps it, and past that only by what every atom keeps (its int16 slot keys,
    their count and its tile's slice flags); the plan does not depend on the atoms; refusals for bad
    sizes and for more intervals per centre type than the shared-memory key map holds."""
    import __graft_entry__
    __graft_entry__._load_builder().build()
    import paper_2107_02103_gb300 as dpc
    info = dpc.dp_table_info_make(0.0, 0.5, 0.01, 0.1, 5.0)   # 50 fine + 20 coarse intervals
    sizes = [dpc.dp_tabulate_tc_work_bytes(info, n, 512, 1, 100) for n in (1, 100, 16416, 40000)]
    assert all(b > 0 and b % 256 == 0 for b in sizes)
    assert sizes[0] <= sizes[1] <= sizes[2] < sizes[3]
    cap, nsl = 70, -(-6 * 70 // 16)                            # slots per atom, K slices
    per_atom = 2 * cap + 4 + nsl / 12                          # keys, count, flags of its tile
    assert abs(sizes[3] - sizes[2] - (40000 - 16416) * per_atom) <= 4 * 256
    assert dpc.dp_tabulate_tc_work_bytes(info, 100, 512, 3, 100) > sizes[1]   # K grows with the types
    for bad in ((info, -1, 512, 1, 100), (info, 10, 0, 1, 100), (info, 10, 512, 9, 100), (info, 10, 512, 1, 0)):
        with pytest.raises(ValueError):
            dpc.dp_tabulate_tc_work_bytes(*bad)
    wide = dpc.dp_table_info_make(0.0, 0.5, 0.0001, 0.1, 5.0)   # 5000 fine intervals
    with pytest.raises(ValueError):
        dpc.dp_tabulate_tc_work_bytes(wide, 10, 512, 1, 100)
    plan = [dpc.dp_tabulate_tc_plan_bytes(info, 512, t, 100) for t in (1, 2, 3)]
    assert all(b > 0 and b % 256 == 0 for b in plan) and plan[0] < plan[1] < plan[2]
    assert dpc.dp_tabulate_tc_plan_bytes(info, 512, 1, 100) == dpc.dp_tabulate_tc_plan_bytes(info, 64, 1, 100)
    for bad in ((info, 0, 1, 100), (info, 512, 9, 100), (info, 512, 1, 0), (wide, 512, 1, 100)):
        with pytest.raises(ValueError):
            dpc.dp_tabulate_tc_plan_bytes(*bad)
