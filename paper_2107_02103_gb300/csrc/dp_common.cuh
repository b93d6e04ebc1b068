// Internal declarations shared by the library's translation units: error
// state, table geometry, the interval search, and small load helpers.
#pragma once

#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "dp_compress.h"
#include "dp_df64.cuh"

namespace dpc {

using dfl::df64;

// ---------------------------------------------------------------- errors
int set_error(int code, const char *fmt, ...);  // stores the message, returns code
void clear_error();
int launch_status(const char *what);  // DP_ERR_CUDA if the last launch failed
void prof_mark(const char *name, cudaStream_t st);  // kernel timing hook (dp_profile_begin)
int take_wait_timeouts_tabulate(unsigned int *count);  // GEMM wait timeouts per unit (dp_tc_wait_timeouts)
int take_wait_timeouts_fitting(unsigned int *count);

// --------------------------------------------------------- table geometry
// dp_table_info with its derived sizes and reciprocal steps.
struct TableGeom {
  double lower, upper, upper_ext, stride0, stride1, inv0, inv1;
  int32_t n0, n1, nint;
};

int make_geom(const dp_table_info *info, TableGeom *g);  // validates; DP_ERR_TABLE_INFO / DP_ERR_NULL

// Per-type row layout: sel[b] rows of type b starting at off[b].
struct Segments {
  int32_t ntypes, nnei;
  int32_t sel[DP_MAX_TYPES];
};
int make_segments(int ntypes, const int32_t *sel, int nnei, Segments *out);

// Node x_l of the grid (Sec. II, the interpolation points): fine nodes
// lower + l*stride0, the junction node `upper`, coarse nodes upper + k*stride1.
__host__ __device__ __forceinline__ double node_x(const TableGeom &g, int l) {
  if (l < g.n0) return g.lower + (double)l * g.stride0;
  if (l == g.n0) return g.upper;
  return g.upper + (double)(l - g.n0) * g.stride1;
}

// Interval l of input s and local variable t = s - x_l (Sec. II: g_m^l is a
// polynomial in the offset from the left node of its interval).
//   lower <= s < upper      -> l = floor((s - lower)/stride0) kept in [0, n0)
//   upper <= s < upper_ext  -> l = n0 + floor((s - upper)/stride1) kept in [n0, nint)
//   s < lower               -> first node (l = 0, t = 0), clamped
//   s >= upper_ext          -> last node (l = nint-1, t = its width), clamped
//   s NaN                   -> l = 0, t = NaN (propagates into the results)
// Clamped inputs see the end value of the table and a zero derivative.
__device__ __forceinline__ int locate(const TableGeom &g, double s, double &t, bool &clamped) {
  clamped = false;
  if (s >= g.lower) {
    if (s < g.upper) {
      const int l = min((int)((s - g.lower) * g.inv0), g.n0 - 1);
      t = s - node_x(g, l);
      return l;
    }
    if (s < g.upper_ext) {
      const int k = min((int)((s - g.upper) * g.inv1), g.n1 - 1);
      t = s - node_x(g, g.n0 + k);
      return g.n0 + k;
    }
    clamped = true;
    t = g.n1 > 0 ? g.stride1 : g.stride0;
    return g.nint - 1;
  }
  if (s < g.lower) {
    clamped = true;
    t = 0.0;
    return 0;
  }
  t = s;  // NaN
  return 0;
}

// The same grid and search in f32 arithmetic, for the f32 kernels: there the
// FP64 pipe is 64x slower than the FFMA pipe, so even a per-neighbour double
// search would cost as much as the channel work it serves.  The oracle runs
// the search in double on the same f32 inputs; the two can differ only at a
// node (where both intervals give the same value, the table being C2) and by
// the f32 rounding of t (~1e-7 absolute), far inside the f32 tolerance.
struct TableGeomF {
  float lower, upper, upper_ext, stride0, stride1, inv0, inv1;
  int32_t n0, n1, nint;
};

inline TableGeomF to_f32(const TableGeom &g) {
  TableGeomF f;
  f.lower = (float)g.lower;
  f.upper = (float)g.upper;
  f.upper_ext = (float)g.upper_ext;
  f.stride0 = (float)g.stride0;
  f.stride1 = (float)g.stride1;
  f.inv0 = (float)g.inv0;
  f.inv1 = (float)g.inv1;
  f.n0 = g.n0;
  f.n1 = g.n1;
  f.nint = g.nint;
  return f;
}

__device__ __forceinline__ int locate(const TableGeomF &g, float s, float &t, bool &clamped) {
  clamped = false;
  if (s >= g.lower) {
    if (s < g.upper) {
      const int l = min((int)((s - g.lower) * g.inv0), g.n0 - 1);
      t = s - fmaf((float)l, g.stride0, g.lower);
      return l;
    }
    if (s < g.upper_ext) {
      const int k = min((int)((s - g.upper) * g.inv1), g.n1 - 1);
      t = s - fmaf((float)k, g.stride1, g.upper);
      return g.n0 + k;
    }
    clamped = true;
    t = g.n1 > 0 ? g.stride1 : g.stride0;
    return g.nint - 1;
  }
  if (s < g.lower) {
    clamped = true;
    t = 0.0f;
    return 0;
  }
  t = s;  // NaN
  return 0;
}

// df64 kernels search in double (one search per neighbour row, off the FP32
// pipes that carry their arithmetic) and split t into a df64.
__device__ __forceinline__ int locate(const TableGeom &g, double s, df64 &t, bool &clamped) {
  double td;
  const int l = locate(g, s, td, clamped);
  t = dfl::split(td);
  return l;
}

// Geometry type used by the kernels of each arithmetic.
template <typename real> struct GeomOf;
template <> struct GeomOf<double> {
  using type = TableGeom;
  static TableGeom make(const TableGeom &g) { return g; }
};
template <> struct GeomOf<float> {
  using type = TableGeomF;
  static TableGeomF make(const TableGeom &g) { return to_f32(g); }
};
template <> struct GeomOf<df64> {
  using type = TableGeom;
  static TableGeom make(const TableGeom &g) { return g; }
};

// Element type of the arrays a kernel of arithmetic `real` reads and writes
// (s, R~, dE/dT, T, ds, dR~): the arithmetic type itself, except df64
// kernels, which take and return double.  Tables are stored in the
// arithmetic type (a df64 table holds (hi, lo) float pairs).
template <typename real> constexpr bool is_df64 = false;
template <> constexpr bool is_df64<df64> = true;

template <typename real> struct IoOf { using type = real; };
template <> struct IoOf<df64> { using type = double; };
template <typename real>
using io_t = typename IoOf<real>::type;

__device__ __forceinline__ double to_io(const double x) { return x; }
__device__ __forceinline__ float to_io(const float x) { return x; }
__device__ __forceinline__ double to_io(const df64 x) { return dfl::join(x); }

template <typename real>
__device__ __forceinline__ real from_io(const io_t<real> x) { return x; }
template <>
__device__ __forceinline__ df64 from_io<df64>(const double x) { return dfl::split(x); }

// A double in the arithmetic type, on the device (table coefficients).
template <typename real>
__device__ __forceinline__ real dcvt(const double x) { return (real)x; }
template <>
__device__ __forceinline__ df64 dcvt<df64>(const double x) { return dfl::from_double(x); }

// A host-side double in the arithmetic type (kernel parameters).
template <typename real>
inline real host_cvt(const double x) { return (real)x; }
template <>
inline df64 host_cvt<df64>(const double x) { return dfl::from_double(x); }

// Warp shuffles of one value of any arithmetic type (a df64 moves as two floats).
__device__ __forceinline__ double shfl(const double v, const int src) { return __shfl_sync(0xffffffffu, v, src); }
__device__ __forceinline__ float shfl(const float v, const int src) { return __shfl_sync(0xffffffffu, v, src); }
__device__ __forceinline__ df64 shfl(const df64 v, const int src) {
  return df64(__shfl_sync(0xffffffffu, v.hi, src), __shfl_sync(0xffffffffu, v.lo, src));
}
__device__ __forceinline__ double shfl_xor(const double v, const int m) { return __shfl_xor_sync(0xffffffffu, v, m); }
__device__ __forceinline__ float shfl_xor(const float v, const int m) { return __shfl_xor_sync(0xffffffffu, v, m); }
__device__ __forceinline__ df64 shfl_xor(const df64 v, const int m) {
  return df64(__shfl_xor_sync(0xffffffffu, v.hi, m), __shfl_xor_sync(0xffffffffu, v.lo, m));
}

// ------------------------------------------------------- vector helpers
template <typename real> struct Vec4;
template <> struct Vec4<double> {
  double x, y, z, w;
};
template <> struct Vec4<float> {
  float x, y, z, w;
};
template <> struct Vec4<df64> {
  df64 x, y, z, w;
};

// Four consecutive values (an environment-matrix row, a dT column).
__device__ __forceinline__ Vec4<double> ld4(const double *p) {
  const double2 a = __ldg(reinterpret_cast<const double2 *>(p));
  const double2 b = __ldg(reinterpret_cast<const double2 *>(p) + 1);
  return {a.x, a.y, b.x, b.y};
}
__device__ __forceinline__ Vec4<float> ld4(const float *p) {
  const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
  return {a.x, a.y, a.z, a.w};
}
// Four consecutive I/O values in the arithmetic type `real`.
template <typename real>
__device__ __forceinline__ Vec4<real> ld4r(const io_t<real> *p) { return ld4(p); }
template <>
__device__ __forceinline__ Vec4<df64> ld4r<df64>(const double *p) {
  const Vec4<double> v = ld4(p);
  return {dfl::split(v.x), dfl::split(v.y), dfl::split(v.z), dfl::split(v.w)};
}

// The six coefficients (a, b, c, d, e, f) of channel m of one interval.  An
// interval's block of 6*M1 values is stored pair-planar, [3][M1][2]: the
// (a, b) pairs of all channels, then the (c, d) pairs, then the (e, f) pairs.
// Lanes that read consecutive channels then read consecutive 2-vectors: each
// of the three loads of a warp is fully coalesced (no sector fetched twice).
__device__ __forceinline__ void ld6(const double *blk, int M1, int m, double c[6]) {
  const double2 *q = reinterpret_cast<const double2 *>(blk) + m;
  const double2 x = __ldg(q), y = __ldg(q + M1), z = __ldg(q + 2 * M1);
  c[0] = x.x; c[1] = x.y; c[2] = y.x; c[3] = y.y; c[4] = z.x; c[5] = z.y;
}
__device__ __forceinline__ void ld6(const float *blk, int M1, int m, float c[6]) {
  const float2 *q = reinterpret_cast<const float2 *>(blk) + m;
  const float2 x = __ldg(q), y = __ldg(q + M1), z = __ldg(q + 2 * M1);
  c[0] = x.x; c[1] = x.y; c[2] = y.x; c[3] = y.y; c[4] = z.x; c[5] = z.y;
}

// df64 table: the (a, b) pair of a channel is one 16-byte (a.hi, a.lo, b.hi, b.lo) vector.
__device__ __forceinline__ void ld6(const df64 *blk, int M1, int m, df64 c[6]) {
  const float4 *q = reinterpret_cast<const float4 *>(blk) + m;
  const float4 x = __ldg(q), y = __ldg(q + M1), z = __ldg(q + 2 * M1);
  c[0] = df64(x.x, x.y); c[1] = df64(x.z, x.w); c[2] = df64(y.x, y.y);
  c[3] = df64(y.z, y.w); c[4] = df64(z.x, z.y); c[5] = df64(z.z, z.w);
}

__device__ __forceinline__ void st4(double *p, double a, double b, double c, double d) {
  reinterpret_cast<double2 *>(p)[0] = make_double2(a, b);
  reinterpret_cast<double2 *>(p)[1] = make_double2(c, d);
}
__device__ __forceinline__ void st4(float *p, float a, float b, float c, float d) {
  *reinterpret_cast<float4 *>(p) = make_float4(a, b, c, d);
}
__device__ __forceinline__ void st4(double *p, df64 a, df64 b, df64 c, df64 d) {
  st4(p, to_io(a), to_io(b), to_io(c), to_io(d));
}

__device__ __forceinline__ int clampi(int x, int lo, int hi) { return min(max(x, lo), hi); }

// Validation shared by the forward and gradient entry points.
int check_fusion_args(const void *table, const dp_table_info *info, const void *s, const void *Rt, int64_t nloc,
                      int nnei, int ntypes, const int32_t *sel, int M1, const void *out0, const void *out1,
                      TableGeom *g, Segments *seg);

}  // namespace dpc
