"""Seeded input generator: determinism, geometry and neighbour-list invariants (CPU only)."""
import math

import numpy as np
import pytest

import workloads as W


def test_deterministic_functions():
    lib = W._get_lib()
    for x in (1e-300, 0.001, 0.5, 1.0, 2.0, 3.7, 1e10):
        assert abs(lib.wl_det_log(x) - math.log(x)) <= 4e-16 * max(1.0, abs(math.log(x)))
    for x in np.linspace(0.0, math.pi, 37):
        assert abs(lib.wl_det_cos(float(x)) - math.cos(x)) <= 4e-16


def test_normal_moments_and_seed():
    a = W.normal(123, (200000,))
    b = W.normal(123, (200000,))
    c = W.normal(124, (200000,))
    assert np.array_equal(a, b) and not np.array_equal(a, c)
    assert abs(a.mean()) < 0.01 and abs(a.std() - 1.0) < 0.01


def test_switch_function():
    rcs, rc = 0.5, 4.0
    assert W.switch(0.3, rcs, rc) == pytest.approx(1 / 0.3, rel=1e-15)
    assert W.switch(4.0, rcs, rc) == 0.0 and W.switch(5.0, rcs, rc) == 0.0
    r = 2.0
    exp = (0.5 * math.cos(math.pi * (r - rcs) / (rc - rcs)) + 0.5) / r
    assert W.switch(r, rcs, rc) == pytest.approx(exp, rel=1e-14)
    u = (r - rcs) / (rc - rcs)
    assert W.switch(r, rcs, rc, 1) == pytest.approx((u ** 3 * (-6 * u * u + 15 * u - 10) + 1) / r, rel=1e-14)


def _rows_ok(w):
    nnei = w.nnei
    off = np.concatenate([[0], np.cumsum(w.sel)])
    assert w.s.shape == (w.nloc, nnei) and w.Rt.shape == (w.nloc, nnei, 4)
    assert np.all(w.nvalid >= 0) and np.all(w.nvalid <= w.sel[None, :])
    for b in range(w.ntypes):
        seg = slice(off[b], off[b + 1])
        valid = np.arange(w.sel[b])[None, :] < w.nvalid[:, b:b + 1]
        assert np.all(w.s[:, seg][~valid] == 0.0) and np.all(w.Rt[:, seg][~valid] == 0.0)
        sv = np.where(valid, w.s[:, seg], 0.0)
        # sorted by distance -> s non-increasing within the valid part of a segment
        d = np.diff(sv, axis=1)
        both = valid[:, 1:]
        assert np.all(d[both] <= 1e-15)
    assert np.array_equal(w.s, w.Rt[..., 0])
    norm = np.linalg.norm(w.Rt[..., 1:], axis=-1)
    assert np.allclose(norm, np.abs(w.s), rtol=1e-13, atol=0)


def test_tiny():
    w = W.make("tiny")
    assert (w.nloc, w.nnei, w.M1, w.M2) == (64, 32, 32, 4)
    assert np.all(w.nvalid == 24)
    _rows_ok(w)
    assert np.array_equal(W.make("tiny").Rt, w.Rt)


def _brute_force_rows(w, rc, rcs):
    """Neighbour rows of every atom by an O(N^2) minimum-image scan (numpy), as (s, R~, nvalid)."""
    pos, box = w.pos, w.box
    nnei = w.nnei
    off = np.concatenate([[0], np.cumsum(w.sel)])
    s = np.zeros((w.nloc, nnei))
    Rt = np.zeros((w.nloc, nnei, 4))
    nvalid = np.zeros((w.nloc, w.ntypes), np.int32)
    for i in range(w.nloc):
        d = pos - pos[i]
        d -= box * np.round(d / box)
        r = np.linalg.norm(d, axis=1)
        r[i] = np.inf
        for b in range(w.ntypes):
            idx = np.where((r < rc) & (w.atype == b))[0]
            idx = idx[np.lexsort((idx, r[idx]))][: w.sel[b]]
            nvalid[i, b] = idx.size
            for q, j in enumerate(idx):
                sv = W.switch(r[j], rcs, rc)
                s[i, off[b] + q] = sv
                Rt[i, off[b] + q] = [sv, sv * d[j, 0] / r[j], sv * d[j, 1] / r[j], sv * d[j, 2] / r[j]]
    return s, Rt, nvalid


def test_water_small_against_brute_force():
    w = W.water(seed=9, nmol=48, sel=(30, 60), rc=5.0)
    _rows_ok(w)
    assert w.atype[:48].tolist() == [0] * 48 and np.all(w.atype[48:] == 1)
    s, Rt, nvalid = _brute_force_rows(w, 5.0, 0.5)
    assert np.array_equal(nvalid, w.nvalid)
    assert np.allclose(s, w.s, rtol=1e-13, atol=1e-16) and np.allclose(Rt, w.Rt, rtol=1e-12, atol=1e-15)
    # every O sees its own two H at r_oh = 0.96
    assert np.allclose(w.s[:48, 30:32], W.switch(0.96, 0.5, 5.0), rtol=1e-9)


def test_fcc_against_brute_force_and_density():
    w = W.cu(seed=5, cells=(6, 6, 6), fill=0.5, sel=160)
    _rows_ok(w)
    s, Rt, nvalid = _brute_force_rows(w, 8.0, 2.0)
    assert np.array_equal(nvalid, w.nvalid)
    assert np.allclose(Rt, w.Rt, rtol=1e-12, atol=1e-15)
    exp = 0.5 * 160  # 4 atoms per a^3 inside the cutoff sphere
    assert abs(w.nvalid.mean() - exp) < 0.04 * exp


@pytest.mark.parametrize("name,kw,fill", [("cu85", {}, 0.83), ("water", {}, 0.65)])
def test_paper_sized_workloads(name, kw, fill):
    w = W.make(name, **kw)
    _rows_ok(w)
    assert abs(w.fill - fill) < 0.02
    assert w.stats["rows_dropped_by_sel"] == 0


def test_shard_partition():
    for n, world in ((10, 3), (4096, 8), (1, 2), (0, 2)):
        spans = [W.shard(n, r, world) for r in range(world)]
        assert spans[0][0] == 0 and spans[-1][1] == n
        assert all(spans[r][1] == spans[r + 1][0] for r in range(world - 1))
        assert max(b - a for a, b in spans) - min(b - a for a, b in spans) <= 1
