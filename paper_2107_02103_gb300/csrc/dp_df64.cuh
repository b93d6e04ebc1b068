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

}  // namespace dfl
}  // namespace dpc
