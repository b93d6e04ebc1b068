// Double-float ("df64") arithmetic on the FP32 pipes.
//
// A df64 value is the unevaluated sum hi + lo of two floats, |lo| of the
// order of an ulp of hi: 48 significant bits, the exponent range of float.
// GB300 retires FP64 at 2 lanes per clock per SM but FP32 at 128, so a
// product-and-accumulate in df64 -- twelve FP32 instructions, built from
// the error-free transformations below -- runs about five times faster
// than the same operation in hardware FP64.  The tabulate-fusion sums are
// long dot products of O(1) values; in df64 their error stays near
// n * 2^-48 of the largest partial sum, a few 1e-13 for the sums here.
//
// Error-free transformations (exact for finite floats, no overflow):
//   two_prod(a, b) = (p, e): p = fl(a b), e = a b - p exactly (one FMA);
//   two_sum(a, b)  = (s, e): s = fl(a + b), e = a + b - s exactly (Knuth's
//                    six-operation form, no condition on the magnitudes).
// The intrinsics below are never contracted or reassociated by the
// compiler, which the transformations rely on.
//
// Results are left "nearly normalised": lo collects the exact errors and the
// small cross terms without a final renormalisation.  A value is only ever
// consumed by another df64 operation or converted to double (hi + lo in
// double, exact up to one rounding), so the normalisation is not needed.
#pragma once

#include <cuda_runtime.h>

namespace dpc {
namespace dfl {

struct df64 {
  float hi, lo;
  df64() = default;
  __host__ __device__ constexpr explicit df64(float h, float l = 0.0f) : hi(h), lo(l) {}
};

// a b + c: exact product of the high parts, the two cross terms (their
// rounding is 2^-48 relative), exact sum of the high parts, and the lows.
__device__ __forceinline__ df64 fma(const df64 a, const df64 b, const df64 c) {
  const float p = __fmul_rn(a.hi, b.hi);
  float pe = __fmaf_rn(a.hi, b.hi, -p);
  pe = __fmaf_rn(a.hi, b.lo, pe);
  pe = __fmaf_rn(a.lo, b.hi, pe);
  const float s = __fadd_rn(p, c.hi);
  const float v = __fsub_rn(s, p);
  const float e = __fadd_rn(__fsub_rn(p, __fsub_rn(s, v)), __fsub_rn(c.hi, v));
  return df64(s, __fadd_rn(e, __fadd_rn(pe, c.lo)));
}

__device__ __forceinline__ df64 operator*(const df64 a, const df64 b) {
  const float p = __fmul_rn(a.hi, b.hi);
  float pe = __fmaf_rn(a.hi, b.hi, -p);
  pe = __fmaf_rn(a.hi, b.lo, pe);
  pe = __fmaf_rn(a.lo, b.hi, pe);
  return df64(p, pe);
}

__device__ __forceinline__ df64 operator+(const df64 a, const df64 b) {
  const float s = __fadd_rn(a.hi, b.hi);
  const float v = __fsub_rn(s, a.hi);
  const float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, v)), __fsub_rn(b.hi, v));
  return df64(s, __fadd_rn(e, __fadd_rn(a.lo, b.lo)));
}

__device__ __forceinline__ df64 &operator+=(df64 &a, const df64 b) { return a = a + b; }
__device__ __forceinline__ df64 &operator*=(df64 &a, const df64 b) { return a = a * b; }

// double -> df64: hi = the double rounded to float, lo = the rest rounded to float
__host__ __device__ __forceinline__ df64 from_double(const double x) {
  const float h = (float)x;
  return df64(h, (float)(x - (double)h));
}

__host__ __device__ __forceinline__ double to_double(const df64 a) { return (double)a.hi + (double)a.lo; }

// The same two conversions for the kernels, by integer operations on the bit
// patterns only.  Conversion instructions between float and double execute on
// GB300's FP64 pipe (64 cycles per warp instruction on a sub-partition), and
// a rare-case fallback to them is if-converted by the compiler into every
// call; so the special cases are integer selects as well.
//
// split: hi = x with its significand cut to 24 bits, lo = the remaining 29
// bits cut to 24: |x - hi - lo| < 2^-47 |x| for 2^-79 <= |x| < 2^128.  Below
// that lo is 0 (|x| < 2^-79: 24 bits kept) and below 2^-126 hi is 0 too; at
// or above 2^128 hi is +-inf, and NaN stays NaN.
__device__ __forceinline__ df64 split(const double x) {
  const unsigned hw = (unsigned)__double2hiint(x), lw = (unsigned)__double2loint(x);
  const unsigned e = (hw >> 20) & 0x7ffu;  // biased double exponent
  const unsigned sign = hw & 0x80000000u;
  const unsigned m23 = ((hw & 0xfffffu) << 3) | (lw >> 29);
  unsigned hb = sign | ((e - 896u) << 23) | m23;              // normal float range: 897 <= e <= 1150
  hb = e < 897u ? sign : hb;                                   // tiny: signed zero
  const unsigned nan = (e == 0x7ffu && ((hw & 0xfffffu) | lw)) ? 0x400000u : 0u;
  hb = e > 1150u ? (sign | 0x7f800000u | nan) : hb;            // huge, inf, NaN
  // bits 28..5 of the low word: an integer below 2^24, made exact as a float from two 12-bit halves
  // (2^23 + h - 2^23 is exact for h < 2^23), then scaled by its weight
  const unsigned r24 = (lw & 0x1fffffffu) >> 5;
  const float ra = __fsub_rn(__uint_as_float(0x4b000000u | (r24 >> 12)), 8388608.0f);
  const float rb = __fsub_rn(__uint_as_float(0x4b000000u | (r24 & 0xfffu)), 8388608.0f);
  const float r = __fmaf_rn(ra, 4096.0f, rb);
  const float scale = __uint_as_float(e - 943u < 207u ? (e - 943u) << 23 : 0u);  // 2^(e-1070); 0 outside
  const float lo = __uint_as_float(__float_as_uint(__fmul_rn(r, scale)) ^ sign);
  return df64(__uint_as_float(hb), lo);
}

// A float widened to double by moving its fields (exact for normal floats);
// zero and subnormals give a signed zero, inf and NaN keep their kind.
__device__ __forceinline__ double widen(const float f) {
  const unsigned b = __float_as_uint(f);
  const unsigned e = (b >> 23) & 0xffu, m = b & 0x7fffffu;
  const unsigned sign = b & 0x80000000u;
  unsigned hw = sign | ((e + 896u) << 20) | (m >> 3), lw = m << 29;
  hw = e == 0xffu ? (sign | 0x7ff00000u | (m >> 3) | (m ? 0x80000u : 0u)) : hw;
  hw = e == 0u ? sign : hw;
  lw = e == 0u ? 0u : lw;
  return __hiloint2double((int)hw, (int)lw);
}

// hi + lo in double: one FP64 add.
__device__ __forceinline__ double join(const df64 a) { return __dadd_rn(widen(a.hi), widen(a.lo)); }

// ---------------------------------------------------------------- functions
// (s, e) with s + e == a + b exactly, for |a| >= |b| (or a == 0): Dekker's fast two-sum.
__device__ __forceinline__ df64 fast_two_sum(const float a, const float b) {
  const float s = __fadd_rn(a, b);
  return df64(s, __fsub_rn(b, __fsub_rn(s, a)));
}

__device__ __forceinline__ df64 operator-(const df64 a) { return df64(-a.hi, -a.lo); }
__device__ __forceinline__ bool operator<(const df64 a, const df64 b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo);
}
__device__ __forceinline__ df64 operator-(const df64 a, const df64 b) { return a + (-b); }

// The float nearest a df64 (up to one rounding).  Results are left unnormalised, and after
// a cancellation the whole value can sit in lo (hi == 0), so a float stand-in is hi + lo.
__device__ __forceinline__ float approx(const df64 a) { return __fadd_rn(a.hi, a.lo); }

// 1 / a: the float reciprocal q0 refined by one Newton-Raphson step whose residual
// e = 1 - a q0 is formed in df64 (q = q0 + q0 e); relative error about 2^-46.
__device__ __forceinline__ df64 rcp(const df64 a) {
  const float q0 = __frcp_rn(approx(a));
  const df64 e = fma(-a, df64(q0), df64(1.0f));
  return fast_two_sum(q0, __fmul_rn(q0, approx(e)));
}

// sqrt(a) for a > 0, after Karp and Markstein: y = a x with x the float 1/sqrt(a), corrected
// by (x / 2)(a - y^2) with the residual formed in df64; relative error about 2^-46.
__device__ __forceinline__ df64 sqrt(const df64 a) {
  const float ah = approx(a);
  const float x = __frsqrt_rn(ah);
  const float y = __fmul_rn(ah, x);
  const df64 r = fma(df64(-y), df64(y), a);
  return fast_two_sum(y, __fmul_rn(__fmul_rn(0.5f, x), approx(r)));
}

// sin(pi u) and cos(pi u) for u in [0, 1] (the cosine switch): with x = u - 1/2,
// sin(pi u) = cos(pi x) and cos(pi u) = -sin(pi x); for |x| > 1/4 the pair comes from
// x' = 1/2 - |x| instead (sin(pi x) = sign(x) cos(pi x'), cos(pi x) = sin(pi x')).  On
// |z| = |pi x| <= pi/4 the Taylor series of sin to z^17 and of cos to z^18 leave terms below
// 2^-52 relative; they are summed by Horner's rule in w = z^2.  The coefficients are
// (-1)^k / (2k+1)! and (-1)^k / (2k)!, and pi, each as the float nearest to it plus the float
// nearest to the rest.
__device__ __forceinline__ void sincospi(const df64 u, df64 *sn, df64 *cs) {
  const df64 x = u + df64(-0.5f);
  const float xa = approx(x);
  const bool flip = fabsf(xa) > 0.25f;
  const bool neg = xa < 0.0f;
  const df64 ax = neg ? -x : x;
  const df64 xr = flip ? df64(0.5f) - ax : ax;  // in [0, 1/4]
  const df64 z = xr * df64(3.1415927e+00f, -8.742278e-08f);
  const df64 w = z * z;
  df64 s = df64(2.8114574e-15f, -1.0462085e-22f);
  s = fma(s, w, df64(-7.6471636e-13f, -1.22007105e-20f));
  s = fma(s, w, df64(1.6059044e-10f, -5.3525265e-18f));
  s = fma(s, w, df64(-2.5052108e-08f, -4.417623e-16f));
  s = fma(s, w, df64(2.7557319e-06f, 3.7935712e-14f));
  s = fma(s, w, df64(-1.984127e-04f, 2.7255969e-12f));
  s = fma(s, w, df64(8.333334e-03f, -4.346172e-10f));
  s = fma(s, w, df64(-1.6666667e-01f, 4.967054e-09f));
  s = fma(s * w, z, z);  // sin(z)
  df64 c = df64(-1.5619207e-16f, -1.5404471e-24f);
  c = fma(c, w, df64(4.7794773e-14f, 7.625444e-22f));
  c = fma(c, w, df64(-1.1470745e-11f, -2.3722077e-19f));
  c = fma(c, w, df64(2.0876756e-09f, 1.1082839e-16f));
  c = fma(c, w, df64(-2.755732e-07f, 7.575112e-15f));
  c = fma(c, w, df64(2.4801588e-05f, -3.406996e-13f));
  c = fma(c, w, df64(-1.3888889e-03f, 3.3631094e-11f));
  c = fma(c, w, df64(4.1666668e-02f, -1.2417635e-09f));
  c = fma(c, w, df64(-0.5f));
  c = fma(c, w, df64(1.0f));  // cos(z)
  // sin(pi x) and cos(pi x) for the signed x
  df64 sx = flip ? c : s, cx = flip ? s : c;
  sx = neg ? -sx : sx;
  *sn = cx;   // sin(pi u) = cos(pi x)
  *cs = -sx;  // cos(pi u) = -sin(pi x)
}

// tanh(x) for a double x, computed in df64 on the FP32 pipes and rounded to double once (relative
// error a few 1e-15; the FP64 pipe runs a handful of instructions per call instead of a whole tanh).
// |x| >= 19.1 gives +-1, what tanh rounds to in double there, |x| < 1e-20 gives x; NaN stays NaN.
// Otherwise, with u = expm1(-2|x|) in (-1, 0], tanh(|x|) = -u / (2 + u): no cancellation for small
// |x|.  expm1(y) for y = -2|x| in (-38.2, 0]: Cody and Waite's reduction y = k ln2 + r with
// k = rint(y / ln2), |r| <~ ln2 / 2, ln2 in three parts whose first two carry 16 significant bits
// (so k times them is exact in float for |k| < 256); expm1(r) = r (1 + r (1/2! + r (1/3! + ...)))
// by its Taylor series to r^13 (the next term is below 2^-50 of the sum); then
// expm1(y) = 2^k expm1(r) + (2^k - 1).  The coefficients 1/n! are each the float nearest to them
// plus the float nearest to the rest.
__device__ __forceinline__ double tanh_d(const double x) {
  const double ax = fabs(x);
  if (!(ax < 19.1)) return x != x ? x : copysign(1.0, x);
  if (ax < 1e-20) return x;  // tanh(x) = x (1 - x^2 / 3 ...); and split keeps all 48 bits only above 2^-79
  const df64 y = split(-2.0 * ax);
  const float kf = rintf(y.hi * 1.44269504f);  // |k| <= 28
  df64 r = y + df64(-kf * 0.69314575f);        // k c1, k c2 exact
  r = r + df64(-kf * 1.4285906e-06f);
  r = r + df64(-kf) * df64(1.619851e-11f);
  df64 q = df64(1.6059044e-10f, -5.3525265e-18f);  // 1/13!
  q = fma(q, r, df64(2.0876756e-09f, 1.1082839e-16f));
  q = fma(q, r, df64(2.5052108e-08f, 4.417623e-16f));
  q = fma(q, r, df64(2.755732e-07f, -7.575112e-15f));
  q = fma(q, r, df64(2.7557319e-06f, 3.7935712e-14f));
  q = fma(q, r, df64(2.4801588e-05f, -3.406996e-13f));
  q = fma(q, r, df64(1.984127e-04f, -2.7255969e-12f));
  q = fma(q, r, df64(1.3888889e-03f, -3.3631094e-11f));
  q = fma(q, r, df64(8.333334e-03f, -4.346172e-10f));
  q = fma(q, r, df64(4.1666668e-02f, -1.2417635e-09f));
  q = fma(q, r, df64(1.6666667e-01f, -4.967054e-09f));
  q = fma(q, r, df64(0.5f));
  q = fma(q, r, df64(1.0f));
  const df64 em = q * r;                                            // expm1(r)
  const float p2 = __uint_as_float((unsigned)(127 + (int)kf) << 23);  // 2^k, k >= -28
  const df64 u = fma(em, df64(p2), df64(p2) + df64(-1.0f));        // expm1(y)
  const df64 t = (-u) * rcp(u + df64(2.0f));
  return copysign(join(t), x);
}

}  // namespace dfl
}  // namespace dpc
