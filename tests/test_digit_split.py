"""The arithmetic behind the f64 GEMMs on the tensor cores (dp_fitting_*_tc_f64 and the tensor-core
tabulation), emulated exactly on the CPU: each operand element is cut into nine balanced 6-bit digits
(in [-32, 32]) against its row's (A) or column's (B) power of two, the 45 digit products with
s + t <= 10 are summed per diagonal as integers, and the result is rebuilt.  The checks are the ones
the kernels rely on: the digits rebuild the 53-bit fixed point exactly, every diagonal sum over a
share of K <= 1792 stays below 2^24 (so fp32 sums of it are exact), digits fit fp16 exactly, and the
result lies within K 2^-49 max|a_i| max|b_j| of the exact dot product (an f64 dot product's bound is
K 2^-53 sum|a b|).  The same for the backward tabulation GEMM's seven balanced 8-bit digits (in
[-128, 128], 55 fractional bits, the 28 products with s + t <= 8, K <= 144, bound K 2^-50).  Plus the
host-side work-size query.  CPU only."""
import math
from fractions import Fraction

import numpy as np
import pytest

S, BITS = 9, 6
FRAC = S * BITS - 1      # fractional bits kept (53)
PAD = S * BITS - FRAC    # the digits stand for 2^(E + PAD) sum_s d_s 64^-s
BIAS = sum(32 * 64 ** k for k in range(S - 1))  # makes the eight low fields digit + 32
MAX_SHARE_K = 1792
# the backward tabulation GEMM's scheme: (digits, bits, fractional bits, bias, largest K, error bound exponent)
SCHEME_9x6 = (S, BITS, FRAC, BIAS, MAX_SHARE_K, -49)
SCHEME_7x8 = (7, 8, 55, sum(128 * 256 ** k for k in range(6)), 144, -50)


def row_exponent(v):
    """E with max |v| < 2^E (v finite), as the split kernels take it from the largest exponent field."""
    m = max(abs(float(x)) for x in v)
    if m == 0.0:
        return -1021
    e = math.frexp(m)[1]      # m = f 2^e, 0.5 <= f < 1, so m < 2^e
    return max(e, -1021)


def digits(x, E, scheme=SCHEME_9x6):
    """The balanced base-2^bits digits of x 2^(frac - E) truncated toward zero: the low fields of the
    fixed point plus the bias, less half the base each, and the top digit (fixed + bias) >> bits (ns - 1)."""
    ns, nb, frac, bias = scheme[:4]
    f = Fraction(x) / Fraction(2) ** E
    assert abs(f) < 1
    fixed = math.trunc(f * 2 ** frac)
    g = fixed + bias
    half = 2 ** (nb - 1)
    low = [((g >> (nb * (ns - s))) & (2 ** nb - 1)) - half for s in range(2, ns + 1)]
    d = [g >> (nb * (ns - 1))] + low
    assert sum(dd * 2 ** (nb * (ns - s)) for s, dd in enumerate(d, 1)) == fixed
    assert all(-half <= dd <= half for dd in d)
    return d


def product(A, B, scheme=SCHEME_9x6):
    """C = A B by the digit scheme, each share of K summed per diagonal in exact integers."""
    ns, nb, frac, bias, share = scheme[:5]
    pad = ns * nb - frac
    n, K = A.shape
    N = B.shape[1]
    E = [row_exponent(A[i]) for i in range(n)]
    F = [row_exponent(B[:, j]) for j in range(N)]
    Ad = np.array([[digits(A[i, k], E[i], scheme) for k in range(K)] for i in range(n)], dtype=object)
    Bd = np.array([[digits(B[k, j], F[j], scheme) for j in range(N)] for k in range(K)], dtype=object)
    C = np.empty((n, N))
    peak = 0
    for i in range(n):
        for j in range(N):
            total = Fraction(0)
            for k0 in range(0, K, share):
                diag = [0] * ns
                for k in range(k0, min(K, k0 + share)):
                    for s in range(ns):
                        for t in range(ns - s):
                            diag[s + t] += Ad[i, k][s] * Bd[k, j][t]
                peak = max(peak, max(abs(d) for d in diag))
                total += sum(Fraction(d, 2 ** (nb * (dd + 2))) for dd, d in enumerate(diag))
            C[i, j] = float(total * Fraction(2) ** (E[i] + F[j] + 2 * pad))
    return C, peak


def test_exactness_bounds_of_the_fp32_diagonal_sums():
    ns, nb, frac, bias, share = SCHEME_7x8[:5]
    assert ns * share * 128 * 128 < 2 ** 24 and share % 16 == 0   # the 7 x 8 scheme's diagonals
    assert 1024 + 256 <= 2 ** 11 and frac >= 53 and bias < 2 ** 48
    for f in (2 ** frac - 1, -(2 ** frac - 1)):
        assert -128 <= (f + bias) >> 48 <= 128
    assert S * MAX_SHARE_K * 32 * 32 < 2 ** 24                   # a diagonal's sum over a share
    assert 1024 + 64 <= 2 ** 11                                  # a digit + 32 + 1024 is an exact fp16 integer
    assert FRAC >= 53                                            # every f64 significand
    assert BIAS < 2 ** 48                                        # the top digit stays in [-32, 32]
    for f in (2 ** FRAC - 1, -(2 ** FRAC - 1)):
        top = (f + BIAS) >> 48
        assert -32 <= top <= 32


@pytest.mark.parametrize("K,scaled,scheme", [(70, False, SCHEME_9x6), (500, False, SCHEME_9x6), (40, True, SCHEME_9x6),
                                             (1900, False, SCHEME_9x6), (100, False, SCHEME_7x8),
                                             (144, False, SCHEME_7x8), (40, True, SCHEME_7x8)])
def test_digit_product_within_its_bound(K, scaled, scheme):
    rng = np.random.default_rng(K)
    A = rng.standard_normal((3, K))
    B = rng.standard_normal((K, 2))
    if scaled:  # rows over many decades, a zero row, a subnormal, zeros inside a row
        A *= 10.0 ** rng.uniform(-30, 30, (3, 1))
        A[0] = 0.0
        A[1, ::3] = 0.0
        A[1, 5] = 5e-310
    C, peak = product(A, B, scheme)
    assert peak < 2 ** 24
    for i in range(A.shape[0]):
        for j in range(B.shape[1]):
            exact = sum(Fraction(A[i, k]) * Fraction(B[k, j]) for k in range(K))
            bound = K * 2.0 ** scheme[5] * np.abs(A[i]).max() * np.abs(B[:, j]).max()
            assert abs(Fraction(C[i, j]) - exact) <= Fraction(bound) + Fraction(abs(float(exact))) * 2 ** -52


def test_the_7x8_bound_is_tight_enough_to_fail_a_dropped_diagonal():
    """The 7 x 8 emulation with its last kept diagonal (s + t = 8) dropped misses the bound on short dot
    products (where the terms' errors cannot cancel much): the bound separates the scheme from that slip."""
    rng = np.random.default_rng(7)
    K = 2
    A = rng.standard_normal((8, K))
    B = rng.standard_normal((K, 1))
    ns, nb, frac, bias, share, eb = SCHEME_7x8
    E = [row_exponent(A[i]) for i in range(A.shape[0])]
    F = row_exponent(B[:, 0])
    worst = 0.0
    for i in range(A.shape[0]):
        Ad = [digits(A[i, k], E[i], SCHEME_7x8) for k in range(K)]
        Bd = [digits(B[k, 0], F, SCHEME_7x8) for k in range(K)]
        diag = [0] * ns
        for k in range(K):
            for s in range(ns - 1):            # s + t <= 5: one diagonal short
                for t in range(ns - 1 - s):
                    diag[s + t] += Ad[k][s] * Bd[k][t]
        got = sum(Fraction(d, 2 ** (nb * (dd + 2))) for dd, d in enumerate(diag)) * Fraction(2) ** (E[i] + F + 2)
        exact = sum(Fraction(A[i, k]) * Fraction(B[k, 0]) for k in range(K))
        bound = K * 2.0 ** eb * np.abs(A[i]).max() * np.abs(B[:, 0]).max()
        worst = max(worst, float(abs(got - exact)) / bound)
    assert worst > 1.0


def test_work_size_query():
    import __graft_entry__
    __graft_entry__._load_builder().build()
    import paper_2107_02103_gb300 as dpc
    w = [1600, 240, 240, 240, 1]
    sizes = [dpc.dp_fitting_tc_work_bytes(w, n) for n in (1, 100, 4096, 20000)]
    assert all(b % 256 == 0 and b > 0 for b in sizes)
    assert sizes == sorted(sizes)
    assert sizes[-1] >= 4 * 20000 * 240 * 8                 # the buffers between layers
    assert dpc.dp_fitting_tc_work_bytes([1600, 240, 100], 10) > 0   # several outputs (a head's weights)
    with pytest.raises(ValueError):
        dpc.dp_fitting_tc_work_bytes([1600, 240, 0], 10)     # an empty output layer
