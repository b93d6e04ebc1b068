// Environment-matrix front end and force / virial back end (Sec. II: the
// weighting function s(r), the 4-vector rows and their normalisation; forces
// and virials from the derivatives of E with respect to atom i and its
// neighbours).
//
// Both kernels run one warp per atom with the lanes over its neighbour rows,
// 32 rows per round: the neighbour list, s and R~ are read and written
// coalesced, the neighbour coordinates are gathered (they stay in L2).  The
// arithmetic per row is a square root, a reciprocal, the switch (a sine and
// cosine for the cosine switch) and a few dozen FMA; both kernels are FP64
// bound in f64, like the fusion kernels around them.  The df64 instances
// (double arrays, double-float arithmetic) take the square root, the
// reciprocal and sin/cos(pi u) from dp_df64.cuh.
#include <cuda_runtime.h>

#include "dp_common.cuh"
#include "env_row.cuh"

namespace dpc {
namespace {

constexpr int kEnvWarps = 4;  // atoms per block

template <typename real>
struct EnvParams {
  const io_t<real> *__restrict__ coord;
  const int32_t *__restrict__ nlist;
  io_t<real> *__restrict__ s;
  io_t<real> *__restrict__ Rt;
  int32_t *__restrict__ nvalid;
  const io_t<real> *__restrict__ ds;
  const io_t<real> *__restrict__ dRt;
  io_t<real> *__restrict__ F;
  io_t<real> *__restrict__ virial;
  int64_t nloc;
  int32_t nnei, ntypes;
  int32_t sel[DP_MAX_TYPES];
  real rcs, rc, inv_width, mean, inv_std, inv_std_all;
  int32_t kind;
};

// Segment (neighbour type) of row q.
template <typename real>
__device__ __forceinline__ int segment_of(const EnvParams<real> &P, int q) {
  int b = 0, lim = P.sel[0];
#pragma unroll
  for (int c = 1; c < DP_MAX_TYPES; ++c)
    if (c < P.ntypes && q >= lim) {
      b = c;
      lim += P.sel[c];
    }
  return b;
}

template <typename real>
__global__ void __launch_bounds__(kEnvWarps * 32) env_mat_kernel(const EnvParams<real> P) {
  const int lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * kEnvWarps + (threadIdx.x >> 5);
  if (i >= P.nloc) return;  // warp-uniform
  // d = r_j - r_i is formed in the arrays' own precision before it enters the arithmetic type:
  // in df64 that keeps its relative accuracy independent of how far the atoms sit from the origin
  const io_t<real> xi = P.coord[3 * i], yi = P.coord[3 * i + 1], zi = P.coord[3 * i + 2];
  int count = 0;  // lane b < ntypes: rows of segment b with a neighbour
  for (int q0 = 0; q0 < P.nnei; q0 += 32) {
    const int q = q0 + lane;
    const int64_t row = i * P.nnei + q;
    const int j = q < P.nnei ? __ldg(P.nlist + row) : -1;
    if (q < P.nnei) {
      real sh = real(0), rx = real(0), ry = real(0), rz = real(0);
      if (j >= 0) {
        const real dx = from_io<real>(P.coord[3 * (int64_t)j] - xi),
                   dy = from_io<real>(P.coord[3 * (int64_t)j + 1] - yi),
                   dz = from_io<real>(P.coord[3 * (int64_t)j + 2] - zi);
        const real r2 = fma(dx, dx, fma(dy, dy, dz * dz));
        const real r = sqrt(r2);
        const real inv_r = recip(r);
        real sv, dsv;
        weight(P, r, inv_r, sv, dsv);
        const real a = sv * inv_r * P.inv_std_all;
        sh = (sv - P.mean) * P.inv_std;
        rx = a * dx;
        ry = a * dy;
        rz = a * dz;
      }
      P.s[row] = to_io(sh);
      st4(P.Rt + row * 4, sh, rx, ry, rz);
    }
    const int b = q < P.nnei ? segment_of(P, q) : 0;
#pragma unroll
    for (int c = 0; c < DP_MAX_TYPES; ++c) {
      if (c >= P.ntypes) break;
      const int n = __popc(__ballot_sync(0xffffffffu, j >= 0 && b == c));
      if (lane == c) count += n;
    }
  }
  if (lane < P.ntypes) P.nvalid[i * P.ntypes + lane] = count;
}

template <typename real>
__device__ __forceinline__ real warp_sum(real v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += shfl_xor(v, o);
  return v;
}

template <typename real>
__global__ void __launch_bounds__(kEnvWarps * 32) force_virial_kernel(const EnvParams<real> P) {
  const int lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * kEnvWarps + (threadIdx.x >> 5);
  if (i >= P.nloc) return;  // warp-uniform
  const io_t<real> xi = P.coord[3 * i], yi = P.coord[3 * i + 1], zi = P.coord[3 * i + 2];
  real f0 = real(0), f1 = real(0), f2 = real(0);  // force on atom i from this lane's rows
  real w[9];
#pragma unroll
  for (int x = 0; x < 9; ++x) w[x] = real(0);
  for (int q0 = 0; q0 < P.nnei; q0 += 32) {
    const int q = q0 + lane;
    const int64_t row = i * P.nnei + q;
    const int j = q < P.nnei ? __ldg(P.nlist + row) : -1;
    if (j >= 0) {
      const real d[3] = {from_io<real>(P.coord[3 * (int64_t)j] - xi), from_io<real>(P.coord[3 * (int64_t)j + 1] - yi),
                         from_io<real>(P.coord[3 * (int64_t)j + 2] - zi)};
      const real r2 = fma(d[0], d[0], fma(d[1], d[1], d[2] * d[2]));
      const real r = sqrt(r2);
      const real inv_r = recip(r);
      real sv, dsv;
      weight(P, r, inv_r, sv, dsv);
      const Vec4<real> gR = ld4r<real>(P.dRt + row * 4);
      const real g0 = from_io<real>(__ldg(P.ds + row)) + gR.x;  // the s column feeds both the table input and R~[0]
      const real p = fma(gR.y, d[0], fma(gR.z, d[1], gR.w * d[2]));
      // g = (g0 s'/(r std) + (s'/r^2 - s/r^3) p / std_all) d + s/(r std_all) dR~_xyz
      const real cd = fma(g0 * dsv, inv_r * P.inv_std, (dsv - sv * inv_r) * inv_r * inv_r * p * P.inv_std_all);
      const real ce = sv * inv_r * P.inv_std_all;
      const real g[3] = {fma(cd, d[0], ce * gR.y), fma(cd, d[1], ce * gR.z), fma(cd, d[2], ce * gR.w)};
      f0 += g[0];
      f1 += g[1];
      f2 += g[2];
      atomicAdd(P.F + 3 * (int64_t)j, to_io(-g[0]));
      atomicAdd(P.F + 3 * (int64_t)j + 1, to_io(-g[1]));
      atomicAdd(P.F + 3 * (int64_t)j + 2, to_io(-g[2]));
#pragma unroll
      for (int a = 0; a < 3; ++a)
#pragma unroll
        for (int b = 0; b < 3; ++b) w[3 * a + b] = fma(-d[a], g[b], w[3 * a + b]);
    }
  }
  f0 = warp_sum(f0);
  f1 = warp_sum(f1);
  f2 = warp_sum(f2);
#pragma unroll
  for (int x = 0; x < 9; ++x) w[x] = warp_sum(w[x]);
  if (lane == 0) {
    atomicAdd(P.F + 3 * i, to_io(f0));
    atomicAdd(P.F + 3 * i + 1, to_io(f1));
    atomicAdd(P.F + 3 * i + 2, to_io(f2));
  }
  if (lane < 9) {
    real v = w[0];
#pragma unroll
    for (int x = 1; x < 9; ++x)
      if (lane == x) v = w[x];
    atomicAdd(P.virial + lane, to_io(v));
  }
}


template <typename real>
void fill_env(EnvParams<real> &P, const dp_env_info *env) {
  P.rcs = host_cvt<real>(env->rcs);
  P.rc = host_cvt<real>(env->rc);
  P.inv_width = host_cvt<real>(1.0 / (env->rc - env->rcs));
  P.mean = host_cvt<real>(env->mean);
  P.inv_std = host_cvt<real>(1.0 / env->std);
  P.inv_std_all = host_cvt<real>(1.0 / env->std_all);
  P.kind = env->kind;
}

template <typename real>
int env_mat(const io_t<real> *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes, const int32_t *sel,
            const dp_env_info *env, io_t<real> *s, io_t<real> *Rt, int32_t *nvalid, void *stream) {
  clear_error();
  if (nloc < 0) return set_error(DP_ERR_SHAPE, "nloc = %lld < 0", (long long)nloc);
  Segments seg;
  int rc = make_segments(ntypes, sel, nnei, &seg);
  if (rc) return rc;
  if ((rc = check_env(env))) return rc;
  if (nloc == 0) return DP_OK;
  if (!coord || !nlist || !s || !Rt || !nvalid) return set_error(DP_ERR_NULL, "dp_env_mat: NULL array");
  const int64_t blocks = (nloc + kEnvWarps - 1) / kEnvWarps;
  if (blocks > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
  EnvParams<real> P{};
  P.coord = coord;
  P.nlist = nlist;
  P.s = s;
  P.Rt = Rt;
  P.nvalid = nvalid;
  P.nloc = nloc;
  P.nnei = nnei;
  P.ntypes = ntypes;
  for (int b = 0; b < DP_MAX_TYPES; ++b) P.sel[b] = seg.sel[b];
  fill_env(P, env);
  env_mat_kernel<real><<<(unsigned)blocks, kEnvWarps * 32, 0, (cudaStream_t)stream>>>(P);
  return launch_status("dp_env_mat");
}

template <typename real>
int force_virial(const io_t<real> *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                 const dp_env_info *env, const io_t<real> *ds, const io_t<real> *dRt, io_t<real> *F,
                 io_t<real> *virial, void *stream) {
  clear_error();
  if (nloc < 0) return set_error(DP_ERR_SHAPE, "nloc = %lld < 0", (long long)nloc);
  if (nall < nloc) return set_error(DP_ERR_SHAPE, "nall = %lld < nloc = %lld", (long long)nall, (long long)nloc);
  if (nnei < 1) return set_error(DP_ERR_SHAPE, "nnei = %d < 1", nnei);
  int rc = check_env(env);
  if (rc) return rc;
  if (!virial || (nall > 0 && !F)) return set_error(DP_ERR_NULL, "dp_force_virial: NULL output");
  if (nloc > 0 && (!coord || !nlist || !ds || !dRt)) return set_error(DP_ERR_NULL, "dp_force_virial: NULL input");
  const int64_t blocks = (nloc + kEnvWarps - 1) / kEnvWarps;
  if (blocks > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
  cudaError_t e = cudaMemsetAsync(virial, 0, 9 * sizeof(io_t<real>), (cudaStream_t)stream);
  if (e == cudaSuccess && nall > 0)
    e = cudaMemsetAsync(F, 0, (size_t)nall * 3 * sizeof(io_t<real>), (cudaStream_t)stream);
  if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_force_virial: %s", cudaGetErrorString(e));
  if (nloc == 0) return DP_OK;
  EnvParams<real> P{};
  P.coord = coord;
  P.nlist = nlist;
  P.ds = ds;
  P.dRt = dRt;
  P.F = F;
  P.virial = virial;
  P.nloc = nloc;
  P.nnei = nnei;
  fill_env(P, env);
  force_virial_kernel<real><<<(unsigned)blocks, kEnvWarps * 32, 0, (cudaStream_t)stream>>>(P);
  return launch_status("dp_force_virial");
}

}  // namespace
}  // namespace dpc

extern "C" {

int dp_env_mat_f64(const double *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes,
                   const int32_t *sel, const dp_env_info *env, double *s, double *Rt, int32_t *nvalid,
                   void *stream) {
  return dpc::env_mat<double>(coord, nlist, nloc, nnei, ntypes, sel, env, s, Rt, nvalid, stream);
}

int dp_env_mat_f32(const float *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes, const int32_t *sel,
                   const dp_env_info *env, float *s, float *Rt, int32_t *nvalid, void *stream) {
  return dpc::env_mat<float>(coord, nlist, nloc, nnei, ntypes, sel, env, s, Rt, nvalid, stream);
}

int dp_force_virial_f64(const double *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                        const dp_env_info *env, const double *ds, const double *dRt, double *F, double *virial,
                        void *stream) {
  return dpc::force_virial<double>(coord, nlist, nloc, nall, nnei, env, ds, dRt, F, virial, stream);
}

int dp_env_mat_df64(const double *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes,
                    const int32_t *sel, const dp_env_info *env, double *s, double *Rt, int32_t *nvalid,
                    void *stream) {
  return dpc::env_mat<dpc::df64>(coord, nlist, nloc, nnei, ntypes, sel, env, s, Rt, nvalid, stream);
}

int dp_force_virial_df64(const double *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                         const dp_env_info *env, const double *ds, const double *dRt, double *F, double *virial,
                         void *stream) {
  return dpc::force_virial<dpc::df64>(coord, nlist, nloc, nall, nnei, env, ds, dRt, F, virial, stream);
}

int dp_force_virial_f32(const float *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                        const dp_env_info *env, const float *ds, const float *dRt, float *F, float *virial,
                        void *stream) {
  return dpc::force_virial<float>(coord, nlist, nloc, nall, nnei, env, ds, dRt, F, virial, stream);
}

}  // extern "C"
