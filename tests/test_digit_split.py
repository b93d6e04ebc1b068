"""The arithmetic behind dp_fitting_*_tc_f64 (the f64 fitting-net GEMMs on the tensor cores),
emulated exactly on the CPU: each operand element is cut into nine balanced 6-bit digits (in
[-32, 32]) against its row's (A) or column's (B) power of two, the 45 digit products with s + t <= 10
are summed per diagonal as integers, and the result is rebuilt.  The checks are the ones the kernels
rely on: the digits rebuild the 53-bit fixed point exactly, every diagonal sum over a share of
K <= 1792 stays below 2^24 (so fp32 sums of it are exact), digits fit fp16 exactly, and the result
lies within K 2^-49 max|a_i| max|b_j| of the exact dot product (an f64 dot product's bound is
K 2^-53 sum|a b|).  Plus the host-side work-size query.  CPU only."""
import math
from fractions import Fraction

import numpy as np
import pytest

S, BITS = 9, 6
FRAC = S * BITS - 1      # fractional bits kept (53)
PAD = S * BITS - FRAC    # the digits stand for 2^(E + PAD) sum_s d_s 64^-s
BIAS = sum(32 * 64 ** k for k in range(S - 1))  # makes the eight low fields digit + 32
MAX_SHARE_K = 1792


def row_exponent(v):
    """E with max |v| < 2^E (v finite), as the split kernels take it from the largest exponent field."""
    m = max(abs(float(x)) for x in v)
    if m == 0.0:
        return -1021
    e = math.frexp(m)[1]      # m = f 2^e, 0.5 <= f < 1, so m < 2^e
    return max(e, -1021)


def digits(x, E):
    """The S balanced base-2^BITS digits of x 2^(FRAC - E) truncated toward zero: the eight low fields of
    the fixed point plus BIAS, less 32 each, and the top digit floor((fixed + BIAS) / 2^48)."""
    f = Fraction(x) / Fraction(2) ** E
    assert abs(f) < 1
    fixed = math.trunc(f * 2 ** FRAC)
    g = fixed + BIAS
    low = [((g >> (BITS * (S - s))) & (2 ** BITS - 1)) - 32 for s in range(2, S + 1)]
    d = [g >> (BITS * (S - 1))] + low
    assert sum(dd * 64 ** (S - s) for s, dd in enumerate(d, 1)) == fixed
    return d


def product(A, B):
    """C = A B by the digit scheme, each share of K summed per diagonal in exact integers."""
    n, K = A.shape
    N = B.shape[1]
    E = [row_exponent(A[i]) for i in range(n)]
    F = [row_exponent(B[:, j]) for j in range(N)]
    Ad = np.array([[digits(A[i, k], E[i]) for k in range(K)] for i in range(n)], dtype=object)
    Bd = np.array([[digits(B[k, j], F[j]) for j in range(N)] for k in range(K)], dtype=object)
    C = np.empty((n, N))
    peak = 0
    for i in range(n):
        for j in range(N):
            total = Fraction(0)
            for k0 in range(0, K, MAX_SHARE_K):
                diag = [0] * S
                for k in range(k0, min(K, k0 + MAX_SHARE_K)):
                    for s in range(S):
                        for t in range(S - s):
                            diag[s + t] += Ad[i, k][s] * Bd[k, j][t]
                peak = max(peak, max(abs(d) for d in diag))
                total += sum(Fraction(d, 2 ** (BITS * (dd + 2))) for dd, d in enumerate(diag))
            C[i, j] = float(total * Fraction(2) ** (E[i] + F[j] + 2 * PAD))
    return C, peak


def test_exactness_bounds_of_the_fp32_diagonal_sums():
    assert S * MAX_SHARE_K * 32 * 32 < 2 ** 24                   # a diagonal's sum over a share
    assert 1024 + 64 <= 2 ** 11                                  # a digit + 32 + 1024 is an exact fp16 integer
    assert FRAC >= 53                                            # every f64 significand
    assert BIAS < 2 ** 48                                        # the top digit stays in [-32, 32]
    for f in (2 ** FRAC - 1, -(2 ** FRAC - 1)):
        top = (f + BIAS) >> 48
        assert -32 <= top <= 32


@pytest.mark.parametrize("K,scaled", [(70, False), (500, False), (40, True), (1900, False)])
def test_digit_product_within_its_bound(K, scaled):
    rng = np.random.default_rng(K)
    A = rng.standard_normal((3, K))
    B = rng.standard_normal((K, 2))
    if scaled:  # rows over many decades, a zero row, a subnormal, zeros inside a row
        A *= 10.0 ** rng.uniform(-30, 30, (3, 1))
        A[0] = 0.0
        A[1, ::3] = 0.0
        A[1, 5] = 5e-310
    C, peak = product(A, B)
    assert peak < 2 ** 24
    for i in range(A.shape[0]):
        for j in range(B.shape[1]):
            exact = sum(Fraction(A[i, k]) * Fraction(B[k, j]) for k in range(K))
            bound = K * 2.0 ** -49 * np.abs(A[i]).max() * np.abs(B[:, j]).max()
            assert abs(Fraction(C[i, j]) - exact) <= Fraction(bound) + Fraction(abs(float(exact))) * 2 ** -52


def test_work_size_query():
    import __graft_entry__
    __graft_entry__._load_builder().build()
    import paper_2107_02103_gb300 as dpc
    w = [1600, 240, 240, 240, 1]
    sizes = [dpc.dp_fitting_tc_work_bytes(w, n) for n in (1, 100, 4096, 20000)]
    assert all(b % 256 == 0 and b > 0 for b in sizes)
    assert sizes == sorted(sizes)
    assert sizes[-1] >= 4 * 20000 * 240 * 8                 # the buffers between layers
    with pytest.raises(ValueError):
        dpc.dp_fitting_tc_work_bytes([1600, 240, 2], 10)     # the output layer must have width 1
