"""Pins of the oracle to facts the paper and the mathematics fix.

Each pin_* function takes an `oracle.Oracle` and raises AssertionError when
the oracle disagrees with something that does NOT come from re-running the
oracle's own formula: closed forms, polynomials the quintic Hermite basis
must reproduce exactly, the Hermite remainder bound on sin(), finite
differences, symmetries of the descriptor (Sec. II: translation, rotation and
permutation symmetry), brute-force hand cases, and library matmuls.
test_oracle_pins.py runs them on the real oracle; test_oracle_mutants.py
runs them on oracle builds with planted mistakes and expects a failure.
"""
from __future__ import annotations

import math

import numpy as np

import workloads as W


def _rel(x, ref):
    x, ref = np.asarray(x, dtype=np.float64), np.asarray(ref, dtype=np.float64)
    scale = np.max(np.abs(ref))
    return float(np.max(np.abs(x - ref)) / (scale if scale > 0 else 1.0))


def _poly_nodes(o, info, coef):
    """Node values of p(x) = sum_k coef[k] x^k, its first and second derivative (numpy polyval)."""
    xs = np.array([o.node_x(info, l) for l in range(info.nint + 1)])
    P = np.polynomial.Polynomial(coef)
    return xs, P(xs), P.deriv(1)(xs), P.deriv(2)(xs), P


# --------------------------------------------------------------- embedding net

def pin_net_skip_wiring(o):
    """All weights 0: every layer outputs tanh(bias) plus its skip, so values are hand-computable.

    widths 1-2-4 (both layers double: u = tanh(b) + (v, v)), 1-3-3 (equal: u = tanh(b) + v),
    1-3-5 (no skip).  d/dx of each output is the number of x's it carries; d2 = 0.
    """
    x = 0.37
    # 1 -> 2 -> 4
    b1 = np.array([0.2, -0.7])
    b2 = np.array([0.1, 0.3, -0.4, 0.9])
    params = np.concatenate([np.zeros(2), b1, np.zeros(8), b2])
    y, dy, d2y = o.net_eval(params, [1, 2, 4], x)
    u1 = np.tanh(b1) + x
    exp = np.tanh(b2) + np.concatenate([u1, u1])
    assert _rel(y, exp) < 1e-15, ("1-2-4", y, exp)
    assert np.allclose(dy, 1.0, rtol=0, atol=1e-15) and np.allclose(d2y, 0.0, atol=1e-15)
    # 1 -> 3 -> 3
    b1 = np.array([0.5, -0.25, 1.5])
    b2 = np.array([-1.0, 0.75, 0.05])
    params = np.concatenate([np.zeros(3), b1, np.zeros(9), b2])
    y, dy, d2y = o.net_eval(params, [1, 3, 3], x)
    exp = np.tanh(b2) + np.tanh(b1)  # first layer 1->3: no skip; second 3->3: skip
    assert _rel(y, exp) < 1e-15, ("1-3-3", y, exp)
    assert np.allclose(dy, 0.0, atol=1e-15)
    # 1 -> 3 -> 5 : no skip anywhere, constant output
    b2 = np.array([0.1, 0.2, 0.3, 0.4, 0.5])
    params = np.concatenate([np.zeros(3), b1, np.zeros(15), b2])
    y, dy, _ = o.net_eval(params, [1, 3, 5], x)
    assert _rel(y, np.tanh(b2)) < 1e-15 and np.allclose(dy, 0.0, atol=1e-15)


def pin_net_single_neuron(o):
    """One tanh neuron: G(x) = tanh(w x + b); values against math.tanh, derivatives against FD of math.tanh."""
    w, b = 1.7, -0.3
    for x in (-0.8, 0.0, 0.45, 1.3):
        y, dy, d2y = o.net_eval(np.array([w, b]), [1, 1], x)
        # widths 1->1 keep the width: u = tanh(z) + x
        assert abs(y[0] - (math.tanh(w * x + b) + x)) < 1e-15
        h = 1e-4
        f = lambda z: math.tanh(w * z + b) + z  # noqa: E731
        fd1 = (f(x + h) - f(x - h)) / (2 * h)
        fd2 = (f(x + h) - 2 * f(x) + f(x - h)) / (h * h)
        assert abs(dy[0] - fd1) < 1e-7, (dy[0], fd1)
        assert abs(d2y[0] - fd2) < 1e-5, (d2y[0], fd2)


def pin_net_derivatives_fd(o):
    """Forward-mode G', G'' of a random 1-8-16-32 net against central differences of G and G'."""
    params = W.net_params(11, [1, 8, 16, 32], 1)[0]
    h = 1e-5
    for x in (0.05, 0.4, 0.93):
        y, dy, d2y = o.net_eval(params, [1, 8, 16, 32], x)
        yp, dyp, _ = o.net_eval(params, [1, 8, 16, 32], x + h)
        ym, dym, _ = o.net_eval(params, [1, 8, 16, 32], x - h)
        assert _rel(dy, (yp - ym) / (2 * h)) < 1e-8
        assert _rel(d2y, (dyp - dym) / (2 * h)) < 1e-8


# ----------------------------------------------------------------- table range

def pin_table_info(o):
    """Range rules on hand cases: lower/upper snapped outward to the steps, coarse segment to 5x upper."""
    info = o.table_info(0.0, 1.05)
    assert (info.lower, info.n0, info.n1) == (0.0, 110, 44)
    assert abs(info.upper - 1.1) < 1e-15 and abs(info.upper_ext - 5.5) < 1e-14
    info = o.table_info(-0.237, 0.42)
    assert abs(info.lower + 0.24) < 1e-15 and abs(info.upper - 0.5) < 1e-15 and info.n0 == 74 and info.n1 == 20
    # node positions
    assert o.node_x(info, 0) == info.lower and o.node_x(info, info.n0) == info.upper
    assert abs(o.node_x(info, 3) - (info.lower + 0.03)) < 1e-15
    assert abs(o.node_x(info, info.n0 + 2) - (info.upper + 0.2)) < 1e-15
    assert abs(o.node_x(info, info.nint) - info.upper_ext) < 1e-14


def pin_locate(o):
    """Interval search on hand cases, both segments, both clamps and NaN."""
    info = o.table_info(0.0, 1.05)  # [0, 1.1) step 0.01, [1.1, 5.5) step 0.1
    l, t, c = o.locate(info, 0.035)
    assert (l, c) == (3, False) and abs(t - 0.005) < 1e-15
    l, t, c = o.locate(info, 0.0)
    assert (l, c) == (0, False) and t == 0.0
    l, t, c = o.locate(info, 1.099)
    assert (l, c) == (109, False) and abs(t - 0.009) < 1e-14
    l, t, c = o.locate(info, 1.1)
    assert (l, c) == (110, False) and abs(t) < 1e-15
    l, t, c = o.locate(info, 2.35)
    assert (l, c) == (122, False) and abs(t - 0.05) < 1e-14
    l, t, c = o.locate(info, -0.5)
    assert (l, t, c) == (0, 0.0, True)
    l, t, c = o.locate(info, 5.5)
    assert (l, c) == (153, True) and abs(t - 0.1) < 1e-15
    l, t, c = o.locate(info, 1e9)
    assert (l, c) == (153, True)
    l, t, c = o.locate(info, float("nan"))
    assert l == 0 and math.isnan(t) and not c


# ----------------------------------------------------------------------- table

def pin_table_nodes(o):
    """Table reproduces y, y', y'' at both ends of every interval (<= 1e-12 relative, max-norm per channel).

    At t = 0 this is exact by construction (f = y, e = y', 2d = y''); at t = Dt it
    holds only when a, b, c follow the closed forms.  Continuity C2 across
    intervals follows.
    """
    params = W.net_params(21, [1, 25, 50, 100], 1)[0]
    for step in (0.01, 0.001):
        info = o.table_info(0.0, 0.45, step, 0.1, 5.0)
        y, dy, d2y = o.nodes(params, [1, 25, 50, 100], info)
        tab = o.table_build(y, dy, d2y, info)
        ref = (y, dy, d2y)
        for l in list(range(0, info.n0, max(1, info.n0 // 40))) + [info.n0 - 1, info.n0, info.nint - 1]:
            Dt = info.stride0 if l < info.n0 else info.stride1
            for order in range(3):
                v0 = o.poly_eval(tab, l, 0.0, order)
                v1 = o.poly_eval(tab, l, Dt, order)
                scale = np.maximum(np.abs(ref[order]).max(axis=0), 1e-300)
                e0 = np.max(np.abs(v0 - ref[order][l]) / scale)
                e1 = np.max(np.abs(v1 - ref[order][l + 1]) / scale)
                assert e0 < 1e-15, (step, l, order, e0)
                assert e1 < 1e-12, (step, l, order, e1)


def pin_table_quintic_exact(o):
    """A degree-5 polynomial is its own quintic Hermite interpolant: reproduced to rounding everywhere."""
    rng = np.random.default_rng(5)
    info = o.table_info(0.0, 0.95, 0.05, 0.1, 3.0)
    for deg in (0, 1, 3, 5):
        coef = rng.normal(size=deg + 1)
        xs, y, dy, d2y, P = _poly_nodes(o, info, coef)
        tab = o.table_build(y[:, None], dy[:, None], d2y[:, None], info)
        for l in range(info.nint):
            Dt = info.stride0 if l < info.n0 else info.stride1
            for frac in (0.13, 0.5, 0.87):
                t = frac * Dt
                v = o.poly_eval(tab, l, t, 0)[0]
                ref = P(xs[l] + t)
                assert abs(v - ref) <= 1e-12 * max(1.0, abs(ref)), (deg, l, frac, v, ref)
                d1 = o.poly_eval(tab, l, t, 1)[0]
                assert abs(d1 - P.deriv(1)(xs[l] + t)) <= 1e-10 * max(1.0, abs(P.deriv(1)(xs[l] + t)))


def pin_table_sin_bound(o):
    """sin(w x + p): midpoint error within the Hermite remainder bound w^6 Dt^6 / 46080, and order 6.

    f - p = f^(6)(xi)/6! t^3 (t - Dt)^3, largest at t = Dt/2; |f^(6)| <= w^6.
    Halving Dt divides the error by about 2^6 = 64.
    """
    om, ph = 10.0, 0.3
    errs = []
    for step in (0.1, 0.05):
        info = o.table_info(0.0, 1.0, step, step * 10, 5.0)
        xs = np.array([o.node_x(info, l) for l in range(info.nint + 1)])
        tab = o.table_build(np.sin(om * xs + ph)[:, None], (om * np.cos(om * xs + ph))[:, None],
                            (-om * om * np.sin(om * xs + ph))[:, None], info)
        e = max(abs(o.poly_eval(tab, l, step / 2, 0)[0] - math.sin(om * (xs[l] + step / 2) + ph))
                for l in range(info.n0))
        bound = om ** 6 * step ** 6 / 46080.0
        assert e <= bound * (1 + 1e-6) + 1e-15, (step, e, bound)
        assert e >= 0.5 * bound, (step, e, bound)  # the bound is attained at the midpoint (sanity)
        errs.append(e)
    ratio = errs[0] / errs[1]
    assert 55.0 < ratio < 70.0, ratio


def pin_compressed_vs_net(o):
    """Table of a real net vs the net itself: error falls ~64x when Dt halves (Sec. III: accuracy vs step)."""
    params = W.net_params(31, [1, 8, 16, 32], 1)[0]
    widths = [1, 8, 16, 32]
    errs = []
    for step in (0.08, 0.04):
        info = o.table_info(0.0, 0.8, step, 0.4, 2.0)
        tab = o.tables(params, widths, info)[0]
        mids = []
        for l in range(info.n0):
            x = o.node_x(info, l) + step / 2
            g = o.poly_eval(tab, l, step / 2, 0)
            y, _, _ = o.net_eval(params, widths, x)
            mids.append(np.max(np.abs(g - y)))
        errs.append(max(mids))
    ratio = errs[0] / errs[1]
    assert 40.0 < ratio < 90.0, (errs, ratio)


# ------------------------------------------------------------------- forward

def _poly_table(o, info, coefs):
    """Table [M][...] whose channel m tabulates polynomial coefs[m] (exact for degree <= 5)."""
    cols = [_poly_nodes(o, info, c) for c in coefs]
    y = np.stack([c[1] for c in cols], axis=1)
    dy = np.stack([c[2] for c in cols], axis=1)
    d2y = np.stack([c[3] for c in cols], axis=1)
    return o.table_build(y, dy, d2y, info), [c[4] for c in cols]


def pin_fwd_brute_force(o):
    """One atom, one real neighbour, two padding rows, M = 1, table of p(x) = 1 + 2x - x^3:
    T[k] = R~[k] p(s) / N_c with N_c = 3, by hand."""
    info = o.table_info(0.0, 0.9, 0.01, 0.1, 5.0)
    tab, polys = _poly_table(o, info, [[1.0, 2.0, 0.0, -1.0]])
    s0 = 0.4321
    s = np.array([[s0, 0.0, 0.0]])
    Rt = np.zeros((1, 3, 4))
    Rt[0, 0] = [s0, 0.3, -0.2, 0.1]
    T = o.fwd(tab[None], info, s, Rt, np.array([[1]], np.int32), None, np.array([3], np.int32))
    p = 1 + 2 * s0 - s0 ** 3
    exp = np.array([s0, 0.3, -0.2, 0.1]) * p / 3.0
    assert _rel(T[0, :, 0], exp) < 1e-14, (T[0, :, 0], exp)


def pin_fwd_constant_G(o):
    """G == c (constant tables, two types): T[k][m] = c_m * sum over valid rows of R~[k] / N_c."""
    w = W.tiny(seed=7, nloc=5, nreal=6, sel=9, widths=(1, 4))
    info = o.table_info(w.s_min, w.s_max)
    consts = [0.5, -1.25, 2.0, 3.5]
    tab, _ = _poly_table(o, info, [[c] for c in consts])
    T = o.fwd(tab[None], info, w.s, w.Rt, w.nvalid, None, w.sel)
    sumR = np.array([w.Rt[i, :w.nvalid[i, 0]].sum(axis=0) for i in range(w.nloc)])
    exp = sumR[:, :, None] * np.array(consts)[None, None, :] / w.nnei
    assert _rel(T, exp) < 1e-14


def _small_water(nmol=40):
    return W.water(seed=13, nmol=nmol, widths=(1, 4, 8, 16), M2=4, sel=(20, 40), rc=4.0, rcs=0.5)


def pin_fwd_vs_explicit_G(o):
    """Fused T equals forming the whole G (every row, padding included) then R~^T G / N_c by matmul.

    Fig. 1(b) against Fig. 1(c): the skip of padded rows changes nothing because their R~ rows are 0.
    """
    w = _small_water()
    info = o.table_info(w.s_min, w.s_max)
    tabs = o.tables(w.params, w.widths, info)
    T = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    G = o.embed_rows(tabs, info, w.s, w.atype, w.sel)
    T2 = np.stack([w.Rt[i].T @ G[i] for i in range(w.nloc)]) / w.nnei
    assert _rel(T, T2) < 1e-13, _rel(T, T2)


def pin_fwd_padding(o):
    """Skipped padding = processed padding (nvalid = sel on the same zero rows); more zero rows only rescale."""
    w = _small_water(24)
    info = o.table_info(w.s_min, w.s_max)
    tabs = o.tables(w.params, w.widths, info)
    T = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    full = np.broadcast_to(w.sel, w.nvalid.shape).astype(np.int32)
    Tf = o.fwd(tabs, info, w.s, w.Rt, full, w.atype, w.sel)
    assert _rel(Tf, T) < 1e-14
    # add 5 zero rows to each segment: N_c grows by 10, T * N_c unchanged
    sel2 = w.sel + 5
    s2 = np.zeros((w.nloc, int(sel2.sum())))
    R2 = np.zeros((w.nloc, int(sel2.sum()), 4))
    s2[:, :w.sel[0]] = w.s[:, :w.sel[0]]
    s2[:, sel2[0]:sel2[0] + w.sel[1]] = w.s[:, w.sel[0]:]
    R2[:, :w.sel[0]] = w.Rt[:, :w.sel[0]]
    R2[:, sel2[0]:sel2[0] + w.sel[1]] = w.Rt[:, w.sel[0]:]
    T2 = o.fwd(tabs, info, s2, R2, w.nvalid, w.atype, sel2)
    assert _rel(T2 * sel2.sum(), T * w.nnei) < 1e-14


def pin_fwd_symmetries(o):
    """Permuting valid neighbours of one type leaves T unchanged; rotating (x,y,z) rotates T's last 3 rows."""
    w = _small_water(24)
    info = o.table_info(w.s_min, w.s_max)
    tabs = o.tables(w.params, w.widths, info)
    T = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    rng = np.random.default_rng(3)
    s2, R2 = w.s.copy(), w.Rt.copy()
    for i in range(w.nloc):
        off = 0
        for b in range(w.ntypes):
            nv = w.nvalid[i, b]
            perm = off + rng.permutation(nv)
            s2[i, off:off + nv] = w.s[i, perm]
            R2[i, off:off + nv] = w.Rt[i, perm]
            off += w.sel[b]
    Tp = o.fwd(tabs, info, s2, R2, w.nvalid, w.atype, w.sel)
    assert _rel(Tp, T) < 1e-13
    Q, _ = np.linalg.qr(rng.normal(size=(3, 3)))
    R3 = w.Rt.copy()
    R3[..., 1:] = w.Rt[..., 1:] @ Q.T
    Tr = o.fwd(tabs, info, w.s, R3, w.nvalid, w.atype, w.sel)
    assert _rel(Tr[:, 0], T[:, 0]) < 1e-13
    assert _rel(Tr[:, 1:], np.einsum("ab,nbm->nam", Q, T[:, 1:])) < 1e-13


# ---------------------------------------------------------------------- grad

def pin_grad_fd(o):
    """dE/ds against central differences of L = <dT, T(s)>; dE/dR~ against the exact linear change."""
    w = _small_water(24)
    info = o.table_info(w.s_min, w.s_max)
    tabs = o.tables(w.params, w.widths, info)
    ds, dRt = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, w.dT)
    def L(s, R, i):  # <dT_i, T_i>: only atom i depends on its own rows
        return float(np.sum(w.dT[i] * o.fwd(tabs, info, s, R, w.nvalid, w.atype, w.sel, atoms=[i])[0]))
    rng = np.random.default_rng(8)
    h = 1e-6
    checked = 0
    for _ in range(12):
        i = int(rng.integers(w.nloc))
        b = int(rng.integers(w.ntypes))
        if w.nvalid[i, b] == 0:
            continue
        r = int(w.sel[:b].sum()) + int(rng.integers(w.nvalid[i, b]))
        sp, sm = w.s.copy(), w.s.copy()
        sp[i, r] += h
        sm[i, r] -= h
        fd = (L(sp, w.Rt, i) - L(sm, w.Rt, i)) / (2 * h)
        # tolerance: relative 1e-8 plus the rounding noise of L divided by the step
        Ti = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, atoms=[i])[0]
        noise = 50 * np.finfo(float).eps * float(np.sum(np.abs(w.dT[i] * Ti))) / h
        assert abs(ds[i, r] - fd) <= 1e-8 * abs(fd) + noise, (i, r, ds[i, r], fd, noise)
        k = int(rng.integers(4))
        Rp = w.Rt.copy()
        Rp[i, r, k] += 0.5
        lin = (L(w.s, Rp, i) - L(w.s, w.Rt, i)) / 0.5
        assert abs(dRt[i, r, k] - lin) <= 1e-10 * max(1.0, abs(lin)), (dRt[i, r, k], lin)
        checked += 1
    assert checked >= 6


def pin_grad_identities(o):
    """<dR~, R~> = <dT, T> (T is linear in R~); grad is linear in dT; padding rows get 0; clamped s get ds = 0."""
    w = _small_water(24)
    info = o.table_info(w.s_min, w.s_max)
    tabs = o.tables(w.params, w.widths, info)
    T = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    ds, dRt = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, w.dT)
    lhs, rhs = float(np.sum(dRt * w.Rt)), float(np.sum(w.dT * T))
    assert abs(lhs - rhs) <= 1e-12 * max(1.0, abs(rhs))
    ds2, dR2 = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, 2.0 * w.dT + 0.5 * w.dT[::-1])
    ds3, dR3 = o.grad(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel, w.dT[::-1])
    assert _rel(ds2, 2.0 * ds + 0.5 * ds3) < 1e-13 and _rel(dR2, 2.0 * dRt + 0.5 * dR3) < 1e-13
    mask = np.zeros(w.s.shape, bool)
    off = 0
    for b in range(w.ntypes):
        mask[:, off:off + w.sel[b]] = np.arange(w.sel[b])[None, :] < w.nvalid[:, b:b + 1]
        off += w.sel[b]
    assert np.all(ds[~mask] == 0.0) and np.all(dRt[~mask] == 0.0)
    assert np.any(ds[mask] != 0.0)
    # push a few valid rows beyond upper_ext and below lower: their ds is exactly 0, dR~ is not
    s2 = w.s.copy()
    rows = np.argwhere(mask)[:6]
    for q, (i, r) in enumerate(rows):
        s2[i, r] = info.upper_ext + 1.0 if q % 2 == 0 else info.lower - 1.0
    ds4, dR4 = o.grad(tabs, info, s2, w.Rt, w.nvalid, w.atype, w.sel, w.dT)
    for i, r in rows:
        assert ds4[i, r] == 0.0 and np.any(dR4[i, r] != 0.0)


def pin_grad_brute_force(o):
    """One atom, two real rows and one padding row, M = 2 channels tabulating random quintics on a
    coarse step (Dt = 0.1, where the t^4, t^5 terms matter): by hand,
    dE/dR~[j][k] = (1/3) sum_m dT[k][m] p_m(s_j),  dE/ds[j] = (1/3) sum_m (sum_k dT[k][m] R~[j][k]) p_m'(s_j)."""
    rng = np.random.default_rng(12)
    info = o.table_info(0.0, 0.95, 0.1, 0.5, 3.0)
    coefs = [rng.normal(size=6) * 3.0, rng.normal(size=6) * 3.0]
    tab, polys = _poly_table(o, info, coefs)
    s = np.array([[0.537, 0.164, 0.0]])
    Rt = np.zeros((1, 3, 4))
    Rt[0, 0] = [0.537, 0.2, -0.4, 0.3]
    Rt[0, 1] = [0.164, -0.1, 0.05, 0.12]
    dT = rng.normal(size=(1, 4, 2))
    ds, dRt = o.grad(tab[None], info, s, Rt, np.array([[2]], np.int32), None, np.array([3], np.int32), dT)
    for j in range(2):
        p = np.array([P(s[0, j]) for P in polys])
        dp = np.array([P.deriv(1)(s[0, j]) for P in polys])
        exp_dR = dT[0] @ p / 3.0
        exp_ds = float(np.sum((dT[0].T @ Rt[0, j]) * dp)) / 3.0
        assert _rel(dRt[0, j], exp_dR) < 1e-12, (dRt[0, j], exp_dR)
        assert abs(ds[0, j] - exp_ds) <= 1e-12 * max(1.0, abs(exp_ds)), (ds[0, j], exp_ds)
    assert ds[0, 2] == 0.0 and np.all(dRt[0, 2] == 0.0)


# ----------------------------------------------------------------- descriptor

def pin_descriptor(o):
    """D = S (S^<)^T against a library matmul; invariant under rotations and same-type permutations."""
    w = _small_water(24)
    info = o.table_info(w.s_min, w.s_max)
    tabs = o.tables(w.params, w.widths, info)
    T = o.fwd(tabs, info, w.s, w.Rt, w.nvalid, w.atype, w.sel)
    D = o.descriptor(T, w.M2)
    ref = np.stack([(T[i].T @ T[i])[:, :w.M2] for i in range(w.nloc)])
    assert _rel(D, ref) < 1e-14
    assert _rel(D[:, :w.M2, :], np.transpose(D[:, :w.M2, :], (0, 2, 1))) < 1e-15
    rng = np.random.default_rng(4)
    Q, _ = np.linalg.qr(rng.normal(size=(3, 3)))
    R3 = w.Rt.copy()
    R3[..., 1:] = w.Rt[..., 1:] @ Q.T
    D3 = o.descriptor(o.fwd(tabs, info, w.s, R3, w.nvalid, w.atype, w.sel), w.M2)
    assert _rel(D3, D) < 1e-13


def pin_descriptor_grad(o):
    """dE/dT of D = S (S^<)^T: exact central differences (D is quadratic), the Euler identity
    <dT, T> = 2 <dD, D>, and the matrix form dS = dD S^< + [dD^T S in the first M2 rows] by matmul."""
    rng = np.random.default_rng(21)
    n, M, M2 = 5, 13, 4
    T = rng.normal(size=(n, 4, M))
    dD = rng.normal(size=(n, M, M2))
    dT = o.descriptor_grad(T, dD)
    L = lambda TT: float(np.sum(dD * o.descriptor(TT, M2)))  # noqa: E731
    assert abs(float(np.sum(dT * T)) - 2.0 * L(T)) <= 1e-12 * max(1.0, abs(L(T)))
    for (a, k, m) in ((0, 0, 0), (1, 2, 3), (2, 3, 12), (4, 1, 7), (3, 0, 4)):
        Tp, Tm = T.copy(), T.copy()
        Tp[a, k, m] += 0.5
        Tm[a, k, m] -= 0.5
        fd = (L(Tp) - L(Tm)) / 1.0
        assert abs(dT[a, k, m] - fd) <= 1e-11 * max(1.0, abs(fd)), (a, k, m, dT[a, k, m], fd)
    for a in range(n):
        S = T[a].T
        dS = dD[a] @ S[:M2]
        dS[:M2] += dD[a].T @ S
        assert _rel(dT[a], dS.T) < 1e-14


# ------------------------------------------------- environment matrix, forces

def pin_switch(o):
    """s(r) at hand-computable points, s'(r) against central differences, and smoothness at rcs and rc.

    u = 1/2 gives w = 1/2 for both switches; u = 1/4 gives 0.896484375 (quintic, exact in binary)
    and (1 + cos(pi/4))/2 (cosine, library cos).  Both switches and their first derivatives are
    continuous at r = rcs and r = rc (the paper's stated purpose of the switch)."""
    rcs, rc = 2.0, 6.0
    for kind in (0, 1):
        v, d = o.switch(1.5, rcs, rc, kind)
        assert abs(v - 1.0 / 1.5) < 1e-15 and abs(d + 1.0 / 2.25) < 1e-15
        v, _ = o.switch(4.0, rcs, rc, kind)  # u = 1/2
        assert abs(v - 0.5 / 4.0) < 1e-15, (kind, v)
        assert o.switch(6.0, rcs, rc, kind) == (0.0, 0.0) and o.switch(7.0, rcs, rc, kind)[0] == 0.0
        for r in (2.3, 3.1, 4.7, 5.9):
            h = 1e-6
            fd = (o.switch(r + h, rcs, rc, kind)[0] - o.switch(r - h, rcs, rc, kind)[0]) / (2 * h)
            assert abs(fd - o.switch(r, rcs, rc, kind)[1]) < 1e-8, (kind, r)
        for r0 in (rcs, rc):  # value and slope continuous
            e = 1e-9
            lo, hi = o.switch(r0 - e, rcs, rc, kind), o.switch(r0 + e, rcs, rc, kind)
            assert abs(lo[0] - hi[0]) < 1e-8 and abs(lo[1] - hi[1]) < 1e-6, (kind, r0, lo, hi)
    assert abs(o.switch(3.0, rcs, rc, 1)[0] - 0.896484375 / 3.0) < 1e-15
    assert abs(o.switch(3.0, rcs, rc, 0)[0] - (0.5 + 0.5 * math.cos(math.pi / 4)) / 3.0) < 1e-15


def pin_env_mat_hand(o):
    """One neighbour at d = (1, 2, 2), r = 3, inside rcs: R~ = (1/3, 1/9, 2/9, 2/9); with the paper's
    normalisation (mean 0.1, std 2, std_all 3) every entry maps as stated; padding rows are zero."""
    coord = np.array([[0.5, -1.0, 2.0], [1.5, 1.0, 4.0], [9.0, 9.0, 9.0]])
    nlist = np.array([[1, -1, -1], [0, 2, -1]], dtype=np.int32)
    s, Rt = o.env_mat(coord, nlist, 4.0, 20.0)
    assert _rel(Rt[0, 0], [1 / 3, 1 / 9, 2 / 9, 2 / 9]) < 1e-15 and s[0, 0] == Rt[0, 0, 0]
    assert not Rt[0, 1:].any() and not s[0, 1:].any() and not Rt[1, 2].any()
    assert _rel(Rt[1, 0], [1 / 3, -1 / 9, -2 / 9, -2 / 9]) < 1e-15  # the reverse pair
    s2, Rt2 = o.env_mat(coord, nlist, 4.0, 20.0, norm=(0.1, 2.0, 3.0))
    assert _rel(Rt2[0, 0], [(1 / 3 - 0.1) / 2, 1 / 27, 2 / 27, 2 / 27]) < 1e-15 and s2[0, 0] == Rt2[0, 0, 0]


def pin_env_mat_matches_generator(o):
    """Rows from coordinates + neighbour list (periodic images as extra coordinates) equal the rows the
    workload generator builds on its own (minimum image, its own series cos) — two independent codes."""
    for w in (W.cu(seed=11, cells=(6, 6, 6), sel=256, fill=0.8, widths=(1, 4)),
              W.water(seed=12, nmol=160, widths=(1, 4), norm=(0.05, 0.1, 0.2))):
        coord, nlist, _ = W.ghost_system(w)
        e = w.env
        s, Rt = o.env_mat(coord, nlist, e["rcs"], e["rc"], e["kind"], e["norm"])
        assert _rel(s, w.s) < 1e-12 and _rel(Rt, w.Rt) < 1e-12, (w.name, _rel(s, w.s), _rel(Rt, w.Rt))


def _cluster(seed, n=36, L=7.0, rc=4.0, types=2, sel=(20, 30)):
    """Non-periodic random cluster with a brute-force neighbour list (type, then distance)."""
    x = W.uniform(seed, (n, 3), 0.0, L)
    t = (np.arange(n) % types).astype(np.int32)
    off = np.concatenate([[0], np.cumsum(sel)])
    nlist = -np.ones((n, int(off[-1])), dtype=np.int32)
    nvalid = np.zeros((n, types), dtype=np.int32)
    for i in range(n):
        d = np.linalg.norm(x - x[i], axis=1)
        for b in range(types):
            js = [j for j in np.argsort(d, kind="stable") if j != i and t[j] == b and d[j] < rc][:sel[b]]
            nlist[i, off[b]:off[b] + len(js)] = js
            nvalid[i, b] = len(js)
    return x, t, nlist, nvalid, np.array(sel, dtype=np.int32)


def _chain_energy(o, x, t, nlist, nvalid, sel, env, params, widths, info, tabs, dD, M2):
    s, Rt = o.env_mat(x, nlist, env[0], env[1], env[2], env[3])
    T = o.fwd(tabs, info, s, Rt, nvalid, t, sel)
    return float(np.sum(dD * o.descriptor(T, M2))), s, Rt, T


def _chain_forces(o, x, t, nlist, nvalid, sel, env, tabs, info, dD, M2):
    E, s, Rt, T = _chain_energy(o, x, t, nlist, nvalid, sel, env, None, None, info, tabs, dD, M2)
    dT = o.descriptor_grad(T, dD)
    ds, dRt = o.grad(tabs, info, s, Rt, nvalid, t, sel, dT)
    F, Wv = o.force_virial(x, nlist, env[0], env[1], ds, dRt, env[2], env[3])
    return E, F, Wv


def _cluster_model(o, seed, kind, norm):
    x, t, nlist, nvalid, sel = _cluster(seed)
    env = (1.5, 4.0, kind, norm)
    s, _ = o.env_mat(x, nlist, *env[:2], kind, norm)
    widths = [1, 4, 8]
    params = W.net_params(seed + 1, widths, 4)
    valid = nlist >= 0
    info = o.table_info(float(s[valid].min()) - 0.05, float(s[valid].max()) + 0.05)
    tabs = o.tables(params, widths, info)
    dD = W.normal(seed + 2, (x.shape[0], 8, 3))
    return x, t, nlist, nvalid, sel, env, tabs, info, dD


def pin_force_fd(o):
    """Forces of E = sum_i <dD_i, D_i> (coordinates -> rows -> table -> T -> D) against central
    differences of E in every coordinate of four atoms, both switches, with and without normalisation."""
    for seed, kind, norm in ((21, 0, None), (22, 1, (0.2, 0.3, 0.25))):
        x, t, nlist, nvalid, sel, env, tabs, info, dD = _cluster_model(o, seed, kind, norm)
        E, F, _ = _chain_forces(o, x, t, nlist, nvalid, sel, env, tabs, info, dD, 3)
        h = 1e-5
        for a in (0, 7, 18, 35):
            for b in range(3):
                xp, xm = x.copy(), x.copy()
                xp[a, b] += h
                xm[a, b] -= h
                Ep = _chain_energy(o, xp, t, nlist, nvalid, sel, env, None, None, info, tabs, dD, 3)[0]
                Em = _chain_energy(o, xm, t, nlist, nvalid, sel, env, None, None, info, tabs, dD, 3)[0]
                fd = -(Ep - Em) / (2 * h)
                assert abs(fd - F[a, b]) <= 1e-6 * max(1.0, np.abs(F).max()), (seed, a, b, fd, F[a, b])


def pin_force_invariants(o):
    """Translation invariance (sum of forces 0), the virial as sum_a r_a (x) F_a for a cluster, and
    rotation covariance (E unchanged, F rotated, W -> R W R^T) — Sec. II's symmetries."""
    x, t, nlist, nvalid, sel, env, tabs, info, dD = _cluster_model(o, 31, 0, None)
    E, F, Wv = _chain_forces(o, x, t, nlist, nvalid, sel, env, tabs, info, dD, 3)
    scale = np.abs(F).max()
    assert np.abs(F.sum(axis=0)).max() < 1e-12 * scale * x.shape[0]
    assert _rel(Wv, np.einsum("ia,ib->ab", x, F)) < 1e-12
    c, sn = math.cos(0.7), math.sin(0.7)
    Rz = np.array([[c, -sn, 0], [sn, c, 0], [0, 0, 1.0]])
    c2, s2 = math.cos(-1.1), math.sin(-1.1)
    Rx = np.array([[1.0, 0, 0], [0, c2, -s2], [0, s2, c2]])
    R = Rz @ Rx
    E2, F2, W2 = _chain_forces(o, x @ R.T, t, nlist, nvalid, sel, env, tabs, info, dD, 3)
    assert abs(E2 - E) <= 1e-12 * max(1.0, abs(E))
    assert _rel(F2, F @ R.T) < 1e-11 and _rel(W2, R @ Wv @ R.T) < 1e-11
    # an energy that is not rotation invariant, E = sum_i <dT_i, T_i> with dT fixed, has a
    # non-symmetric virial; it is still sum_a r_a (x) F_a
    s, Rt = o.env_mat(x, nlist, env[0], env[1], env[2], env[3])
    dT = W.normal(33, (x.shape[0], 4, 8))
    ds, dRt = o.grad(tabs, info, s, Rt, nvalid, t, sel, dT)
    F3, W3 = o.force_virial(x, nlist, env[0], env[1], ds, dRt, env[2], env[3])
    ref = np.einsum("ia,ib->ab", x, F3)
    assert _rel(W3, ref) < 1e-12 and _rel(ref, ref.T) > 1e-3


# ------------------------------------------------------------------ fitting net

def pin_fitting_hand(o):
    """Nets small enough to evaluate by hand with math.tanh: widths (2, 1, 1) is
    E = w_o tanh(D W_1 + b_1) + b_o and dE/dD_k = w_o (1 - tanh^2) W_1[k]; widths (3, 2, 2, 1) with
    W_2 = 0 shows the skip of the equal-width layer: v_2 = tanh(b_2) + v_1."""
    W1, b1, wo, bo = np.array([0.3, -0.7]), 0.2, 1.5, -0.4
    params = np.concatenate([W1, [b1], [wo], [bo]])
    D = np.array([[0.9, 0.25], [-1.2, 0.4]])
    E, dD = o.fitting(params, [2, 1, 1], D)
    for i in range(2):
        z = D[i] @ W1 + b1
        assert abs(E[i] - (wo * math.tanh(z) + bo)) < 1e-15
        assert _rel(dD[i], wo * (1 - math.tanh(z) ** 2) * W1) < 1e-15
    Wa = np.array([[0.1, -0.2], [0.3, 0.05], [-0.6, 0.4]])
    ba, bb, wout, bout = np.array([0.5, -0.1]), np.array([0.7, 0.2]), np.array([2.0, -1.0]), 0.3
    params = np.concatenate([Wa.ravel(), ba, np.zeros(4), bb, wout, [bout]])
    D = np.array([[1.0, -2.0, 0.5]])
    E = o.fitting(params, [3, 2, 2, 1], D, grad=False)
    v1 = np.tanh(D[0] @ Wa + ba)
    v2 = np.tanh(bb) + v1
    assert abs(E[0] - (v2 @ wout + bout)) < 1e-15


def pin_fitting_fd(o):
    """dE_i/dD_i against central differences of E_i (a 40-wide input, three 24-wide hidden layers
    with skips, two centre types), and linearity of the gradient in the upstream weights g."""
    widths = [40, 24, 24, 24, 1]
    params = W.net_params(61, widths, 2)
    D = W.normal(62, (5, 40))
    at = np.array([0, 1, 1, 0, 1], dtype=np.int32)
    E, dD = o.fitting(params, widths, D, at)
    h = 1e-6
    for i in (0, 2, 4):
        for k in (0, 7, 39):
            Dp, Dm = D.copy(), D.copy()
            Dp[i, k] += h
            Dm[i, k] -= h
            fd = (o.fitting(params, widths, Dp, at, grad=False)[i] - o.fitting(params, widths, Dm, at, grad=False)[i]) / (2 * h)
            assert abs(fd - dD[i, k]) <= 1e-8 * max(1.0, np.abs(dD).max()), (i, k, fd, dD[i, k])
    g = np.array([0.5, -2.0, 1.0, 3.0, 0.0])
    _, dDg = o.fitting(params, widths, D, at, g=g)
    assert _rel(dDg, g[:, None] * dD) < 1e-15


def pin_fitting_types(o):
    """Each atom uses its own centre type's parameters: a two-type batch equals two one-type batches."""
    widths = [10, 6, 6, 1]
    params = W.net_params(63, widths, 2)
    D = W.normal(64, (6, 10))
    at = np.array([1, 0, 1, 1, 0, 0], dtype=np.int32)
    E, dD = o.fitting(params, widths, D, at)
    for t in (0, 1):
        sel = at == t
        Et, dDt = o.fitting(params[t], widths, D[sel])
        assert _rel(E[sel], Et) < 1e-15 and _rel(dD[sel], dDt) < 1e-15


def pin_fitting_multi_output(o):
    """A net with several outputs is several scalar nets sharing the hidden layers: output c equals the
    one-output net whose output layer is column c of W_out and b_out[c] (a net pinned above by hand and
    by differences), and the backward weighted by g [n][nout] is sum_c g_c times that net's dE/dD."""
    widths = [12, 8, 8, 5]
    params = W.net_params(65, widths, 2)
    D = W.normal(66, (7, 12))
    at = np.array([0, 1, 1, 0, 1, 0, 0], dtype=np.int32)
    g = W.normal(67, (7, 5))
    E, dD = o.fitting(params, widths, D, at, g=g)
    a = widths[-2]
    nh = params.shape[1] - (a + 1) * widths[-1]  # the hidden layers' parameters
    ref_dD = np.zeros_like(dD)
    for c in range(widths[-1]):
        Wo = params[:, nh:nh + a * widths[-1]].reshape(2, a, widths[-1])[:, :, c]
        bo = params[:, nh + a * widths[-1] + c]
        pc = np.concatenate([params[:, :nh], Wo, bo[:, None]], axis=1)
        Ec, dDc = o.fitting(pc, widths[:-1] + [1], D, at)
        assert _rel(E[:, c], Ec) < 1e-15, c
        ref_dD += g[:, c:c + 1] * dDc
    assert _rel(dD, ref_dD) < 1e-13


# ------------------------------------------------------------ vector and tensor heads

def _rotation():
    c, sn = math.cos(0.7), math.sin(0.7)
    Rz = np.array([[c, -sn, 0], [sn, c, 0], [0, 0, 1.0]])
    c2, s2 = math.cos(-1.1), math.sin(-1.1)
    Rx = np.array([[1.0, 0, 0], [0, c2, -s2], [0, s2, c2]])
    return Rz @ Rx


def _head_chain(o, x, t, nlist, nvalid, sel, env, tabs, info, fparams, fwidths, M2):
    """Coordinates -> R~ -> T -> D -> the fitting net's M outputs a (invariant) and T."""
    s, Rt = o.env_mat(x, nlist, env[0], env[1], env[2], env[3])
    T = o.fwd(tabs, info, s, Rt, nvalid, t, sel)
    a = o.fitting(fparams, fwidths, o.descriptor(T, M2).reshape(x.shape[0], -1), t, grad=False)
    return T, a


def _head_fd(o, head, grad, T, a, dout, h=1e-6):
    """dT and da of L = <dout, head(T, a)> against central differences in a sample of entries."""
    dT, da = grad(T, a, dout)
    L = lambda T_, a_: float(np.sum(dout * head(T_, a_)))
    for i, k, m in ((0, 0, 0), (1, 1, 2), (2, 2, 5), (3, 3, 7), (1, 3, 0)):
        Tp, Tm = T.copy(), T.copy()
        Tp[i, k, m] += h
        Tm[i, k, m] -= h
        fd = (L(Tp, a) - L(Tm, a)) / (2 * h)
        assert abs(fd - dT[i, k, m]) <= 1e-8 * max(1.0, np.abs(dT).max()), (i, k, m, fd, dT[i, k, m])
    for i, m in ((0, 0), (2, 3), (3, 7)):
        ap, am = a.copy(), a.copy()
        ap[i, m] += h
        am[i, m] -= h
        fd = (L(T, ap) - L(T, am)) / (2 * h)
        assert abs(fd - da[i, m]) <= 1e-8 * max(1.0, np.abs(da).max()), (i, m, fd, da[i, m])


def pin_vector_head(o):
    """v = sum_m a_m T[1:4, m]: a one-hot a picks a column of T's last three rows; a numpy matmul on
    random inputs; the backward against differences; and on the whole vector model from coordinates
    (R~ -> T -> D -> fitting net with M outputs -> v) rotating the coordinates rotates v while a, a
    function of the invariant D, stays (the rotation covariance the head exists for)."""
    T = W.normal(71, (4, 4, 8))
    a = W.normal(72, (4, 8))
    for m in (0, 5):
        e = np.zeros((4, 8))
        e[:, m] = 1.0
        assert np.array_equal(o.vector_head(T, e), T[:, 1:4, m])
    assert _rel(o.vector_head(T, a), np.einsum("ikm,im->ik", T[:, 1:4, :], a)) < 1e-15
    _head_fd(o, o.vector_head, o.vector_head_grad, T, a, W.normal(73, (4, 3)))
    x, t, nlist, nvalid, sel, env, tabs, info, _ = _cluster_model(o, 74, 0, None)
    fwidths = [8 * 3, 10, 10, 8]
    fparams = W.net_params(75, fwidths, 2)
    T, a = _head_chain(o, x, t, nlist, nvalid, sel, env, tabs, info, fparams, fwidths, 3)
    R = _rotation()
    T2, a2 = _head_chain(o, x @ R.T, t, nlist, nvalid, sel, env, tabs, info, fparams, fwidths, 3)
    assert _rel(a2, a) < 1e-12
    assert _rel(o.vector_head(T2, a2), o.vector_head(T, a) @ R.T) < 1e-11


def pin_tensor_head(o):
    """A = sum_m a_m t_m t_m^T (t_m = T[1:4, m]): symmetric; a one-hot a gives the outer product
    t_m t_m^T; its trace is sum_m a_m |t_m|^2; a numpy einsum on random inputs; the backward against
    differences with a non-symmetric dE/dA; and A -> R A R^T when the coordinates of the whole tensor
    model rotate."""
    T = W.normal(81, (4, 4, 8))
    a = W.normal(82, (4, 8))
    A = o.tensor_head(T, a)
    assert np.array_equal(A, np.transpose(A, (0, 2, 1)))
    e = np.zeros((4, 8))
    e[:, 3] = 1.0
    assert _rel(o.tensor_head(T, e), np.einsum("ic,id->icd", T[:, 1:4, 3], T[:, 1:4, 3])) < 1e-15
    assert _rel(np.trace(A, axis1=1, axis2=2), np.einsum("im,ikm,ikm->i", a, T[:, 1:4], T[:, 1:4])) < 1e-14
    assert _rel(A, np.einsum("im,icm,idm->icd", a, T[:, 1:4], T[:, 1:4])) < 1e-14
    _head_fd(o, o.tensor_head, o.tensor_head_grad, T, a, W.normal(83, (4, 3, 3)))
    x, t, nlist, nvalid, sel, env, tabs, info, _ = _cluster_model(o, 84, 1, (0.2, 0.3, 0.25))
    fwidths = [8 * 3, 10, 8]
    fparams = W.net_params(85, fwidths, 2)
    T, a = _head_chain(o, x, t, nlist, nvalid, sel, env, tabs, info, fparams, fwidths, 3)
    R = _rotation()
    T2, a2 = _head_chain(o, x @ R.T, t, nlist, nvalid, sel, env, tabs, info, fparams, fwidths, 3)
    assert _rel(o.tensor_head(T2, a2), R @ o.tensor_head(T, a) @ R.T) < 1e-11


ALL_PINS = [pin_net_skip_wiring, pin_net_single_neuron, pin_net_derivatives_fd, pin_table_info, pin_locate,
            pin_table_nodes, pin_table_quintic_exact, pin_table_sin_bound, pin_compressed_vs_net,
            pin_fwd_brute_force, pin_fwd_constant_G, pin_fwd_vs_explicit_G, pin_fwd_padding, pin_fwd_symmetries,
            pin_grad_fd, pin_grad_identities, pin_grad_brute_force, pin_descriptor, pin_descriptor_grad,
            pin_switch, pin_env_mat_hand, pin_env_mat_matches_generator, pin_force_fd, pin_force_invariants,
            pin_fitting_hand, pin_fitting_fd, pin_fitting_types, pin_fitting_multi_output, pin_vector_head,
            pin_tensor_head]
