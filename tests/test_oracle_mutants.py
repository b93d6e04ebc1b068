"""Plant plausible mistakes in copies of the oracle and check that a pin catches each one (CPU only).

Each mutant is the oracle source with one textual change (a dropped term, a
wrong sign, a swapped index, a transposed operand), compiled into a
temporary library.  The real oracle source is never modified.
"""
import os

import pytest

import oracle
import oracle_pins

MUTANTS = [
    ("a: sign of the y' term", "- 6.0L * (p1 + p0) * Dt", "+ 6.0L * (p1 + p0) * Dt"),
    ("b: swapped y' weights", "(14.0L * p1 + 16.0L * p0)", "(16.0L * p1 + 14.0L * p0)"),
    ("c: sign of y''_{l+1}", "(3.0L * q0 - q1)", "(3.0L * q0 + q1)"),
    ("d = y'' instead of y''/2", "out[3] = (double)(q0 / 2.0L);", "out[3] = (double)(q0);"),
    ("h = y1 + y0", "ld h = y1 - y0;", "ld h = y1 + y0;"),
    ("coarse segment uses the fine step", "ld Dt = (ld)(l < in->n0 ? in->stride0 : in->stride1);",
     "ld Dt = (ld)(in->stride0);"),
    ("net: interleaved instead of concatenated skip", "u[o] = h + v[o % a];", "u[o] = h + v[o / 2];"),
    ("net: sign of tanh''", "ld h2 = sech2 * z2 - 2.0L * h * sech2 * z1 * z1;",
     "ld h2 = sech2 * z2 + 2.0L * h * sech2 * z1 * z1;"),
    ("net: skip missing on equal width", "u[o] = h + v[o];", "u[o] = h;"),
    ("range: floor instead of ceil", "out->upper = stride1 * ceil(s_max / stride1);",
     "out->upper = stride1 * floor(s_max / stride1);"),
    ("node: coarse nodes at fine step", "return in->upper + (double)(l - in->n0) * in->stride1;",
     "return in->upper + (double)(l - in->n0) * in->stride0;"),
    ("locate: ceil instead of floor", "k = (int32_t)floor((x - in->lower) / in->stride0);",
     "k = (int32_t)ceil((x - in->lower) / in->stride0);"),
    ("poly: a and b swapped", "return c[0] * t5 + c[1] * t4", "return c[1] * t5 + c[0] * t4"),
    ("fwd: wrong R~ column", "Ti[k * M + m] += Rt[row * 4 + k] * g;", "Ti[k * M + m] += Rt[row * 4 + (k ^ 1)] * g;"),
    ("fwd: 1/N_c dropped", "Ti[q] = Ti[q] / (double)nnei;", "Ti[q] = Ti[q];"),
    ("fwd: type-segment offset dropped", "int64_t row = i * nnei + off[beta] + j;", "int64_t row = i * nnei + j;"),
    ("grad: g' with 4a t^4", "return 5.0 * c[0] * t4 + 4.0 * c[1] * t3", "return 4.0 * c[0] * t4 + 4.0 * c[1] * t3"),
    ("grad: ds uses g instead of g'", "dsum += rm * dg;", "dsum += rm * g;"),
    ("grad: r_m from one R~ column", "rm += dTi[k * M + m] * Rt[row * 4 + k];", "rm += dTi[k * M + m] * Rt[row * 4 + 0];"),
    ("grad: dR~ uses g'", "dr[k] += dTi[k * M + m] * g;", "dr[k] += dTi[k * M + m] * dg;"),
    ("grad: padding rows processed",
     "for (int j = 0; j < nvalid[i * ntypes + beta]; ++j) {\n        int r = off[beta] + j;",
     "for (int j = 0; j < sel[beta]; ++j) {\n        int r = off[beta] + j;"),
    ("grad: clamp ignored", "double dg = clamped ? 0.0 : poly_dg(c, t);", "double dg = poly_dg(c, t);"),
    ("descriptor: wrong k on S^<", "v += Ta[k * M + m] * Ta[k * M + q];", "v += Ta[k * M + m] * Ta[((k + 1) % 4) * M + q];"),
    ("descriptor grad: S^< term dropped", "if (m < M2)\n          for (int mp = 0; mp < M; ++mp)",
     "if (m < 0)\n          for (int mp = 0; mp < M; ++mp)"),
    ("descriptor grad: transposed dD", "v += Ga[(size_t)mp * M2 + m] * Ta[k * M + mp];",
     "v += Ga[(size_t)m * M2 + (mp % M2)] * Ta[k * M + mp];"),
    ("switch: sign of dw/du", "dw = -30.0 * u * u * (u - 1.0) * (u - 1.0);", "dw = 30.0 * u * u * (u - 1.0) * (u - 1.0);"),
    ("switch: s' without -w/r^2", "*dsv = dw / ((rc - rcs) * r) - w / (r * r);", "*dsv = dw / ((rc - rcs) * r);"),
    ("switch: cosine of u, not pi u", "w = 0.5 * cos(pi * u) + 0.5;", "w = 0.5 * cos(u) + 0.5;"),
    ("env mat: xyz not divided by r", "Rt[4 * row + 1 + a] = sv * d[a] / r / sa;", "Rt[4 * row + 1 + a] = sv * d[a] / sa;"),
    ("env mat: xyz scaled by std of s", "Rt[4 * row + 1 + a] = sv * d[a] / r / sa;",
     "Rt[4 * row + 1 + a] = sv * d[a] / r / sd;"),
    ("force: s column gradient dropped from the first R~ entry",
     "double v = (ds[row] + dRt[4 * row + 0]) * dsv * d[b] / (r * sd);", "double v = ds[row] * dsv * d[b] / (r * sd);"),
    ("force: reaction on j with the wrong sign", "F[3 * (int64_t)j + b] -= g[b];", "F[3 * (int64_t)j + b] += g[b];"),
    ("force: delta term of d(d/r) dropped", "sv * (dab / r - d[a] * d[b] / (r2 * r))", "sv * (0.0 / r - d[a] * d[b] / (r2 * r))"),
    ("virial: sign", "W[3 * a + b] -= d[a] * g[b];", "W[3 * a + b] += d[a] * g[b];"),
    ("virial: transposed", "W[3 * a + b] -= d[a] * g[b];", "W[3 * a + b] -= d[b] * g[a];"),
    ("fitting: skip missing", "act[off_out + o] = t + (b == a ? act[off_in + o] : 0.0);", "act[off_out + o] = t;"),
    ("fitting: backward skip missing", "for (int k = 0; k < ai; ++k) nxt[k] += cur[k];", "for (int k = 0; k < ai; ++k) nxt[k] += 0.0;"),
    ("fitting: tanh' with the wrong sign", "const double gz = cur[o] * (1.0 - t * t);", "const double gz = cur[o] * (1.0 + t * t);"),
    ("fitting: transposed weights", "for (int k = 0; k < a; ++k) z += act[off_in + k] * W[(size_t)k * b + o];",
     "for (int k = 0; k < a; ++k) z += act[off_in + k] * W[(size_t)o * a + k];"),
    ("fitting: centre type ignored", "const double *pp = params + (size_t)(atype ? atype[i] : 0) * P;", "const double *pp = params;"),
    ("fitting: output weights read transposed", "for (int k = 0; k < a; ++k) e += act[off_in + k] * Wo[(size_t)k * nout + c];",
     "for (int k = 0; k < a; ++k) e += act[off_in + k] * Wo[(size_t)c * a + k];"),
    ("fitting: upstream weights of output 0 only",
     "v += (g ? g[(size_t)i * nout + c] : 1.0) * Wo[(size_t)k * nout + c];",
     "v += (g ? g[(size_t)i * nout] : 1.0) * Wo[(size_t)k * nout + c];"),
    ("vector head: row 0 of T included", "s += a[i * M + m] * T[(i * 4 + 1 + c) * M + m];",
     "s += a[i * M + m] * T[(i * 4 + c) * M + m];"),
    ("vector head grad: one component of dv", "dT[(i * 4 + 1 + c) * M + m] = a[i * M + m] * dv[i * 3 + c];",
     "dT[(i * 4 + 1 + c) * M + m] = a[i * M + m] * dv[i * 3];"),
    ("tensor head: diagonal rows only",
     "s += a[i * M + m] * (T[(i * 4 + 1 + c) * M + m] * T[(i * 4 + 1 + d) * M + m]);",
     "s += a[i * M + m] * (T[(i * 4 + 1 + c) * M + m] * T[(i * 4 + 1 + c) * M + m]);"),
    ("tensor head grad: transposed dA term dropped", "u += (G[3 * c + d] + G[3 * d + c]) * td;",
     "u += (G[3 * c + d] + G[3 * c + d]) * td;"),
    ("tensor head grad: da without the a-free product", "s += G[3 * c + d] * T[(i * 4 + 1 + c) * M + m] * td;",
     "s += G[3 * c + d] * td;"),
]


@pytest.mark.parametrize("desc,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(desc, old, new, tmp_path):
    src = open(oracle._SRC).read()
    assert src.count(old) == 1, f"mutation site not unique or missing: {old!r}"
    msrc = tmp_path / "mutant.c"
    msrc.write_text(src.replace(old, new))
    lib = oracle.build(force=True, src=str(msrc), out=str(tmp_path / "libmutant.so"))
    o = oracle.Oracle(lib)
    failures = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(o)
        except Exception as exc:  # noqa: BLE001 - any failure counts as "caught"
            failures.append((pin.__name__, type(exc).__name__))
    assert failures, f"no pin caught the mutant: {desc}"
    os.remove(lib)
