// The weighting function s(r) of the environment matrix (Sec. II) and its derivative, shared by
// env_force.cu's kernels and the tensor-core tabulation's fused rows (tabulate_tc.cu), so that both form
// the same bits.  P supplies rcs, rc, inv_width = 1 / (rc - rcs) and kind; real is double, float or
// df64.
#pragma once

#include "dp_common.cuh"

namespace dpc {
namespace {

__device__ __forceinline__ double recip(const double x) { return 1.0 / x; }
__device__ __forceinline__ float recip(const float x) { return 1.0f / x; }
__device__ __forceinline__ df64 recip(const df64 x) { return dfl::rcp(x); }
__device__ __forceinline__ void sin_cos_pi(const double u, double *s, double *c) { sincospi(u, s, c); }
__device__ __forceinline__ void sin_cos_pi(const float u, float *s, float *c) { sincospif(u, s, c); }
__device__ __forceinline__ void sin_cos_pi(const df64 u, df64 *s, df64 *c) { dfl::sincospi(u, s, c); }
template <typename real>
__device__ __forceinline__ real half_pi() { return real(1.57079632679489661923); }
template <>
__device__ __forceinline__ df64 half_pi<df64>() { return df64(1.5707964e+00f, -4.371139e-08f); }

// s(r) and ds/dr of the weighting function (Sec. II).  u = (r - rcs)/(rc - rcs);
// kind 1: w = u^3 (-6u^2 + 15u - 10) + 1 (the paper's switch), w' = -30 u^2 (u - 1)^2;
// kind 0: w = cos(pi u)/2 + 1/2, w' = -(pi/2) sin(pi u).  inv_r = 1/r.
template <typename real, typename EP>
__device__ __forceinline__ void weight(const EP &P, real r, real inv_r, real &sv, real &dsv) {
  if (r < P.rcs) {
    sv = inv_r;
    dsv = -inv_r * inv_r;
  } else if (r < P.rc) {
    const real u = (r - P.rcs) * P.inv_width;
    real w, dw;
    if (P.kind == 1) {
      const real u2 = u * u, um = u - real(1);
      w = fma(u2 * u, fma(fma(real(-6), u, real(15)), u, real(-10)), real(1));
      dw = real(-30) * u2 * um * um;
    } else {
      real sn, cs;
      sin_cos_pi(u, &sn, &cs);
      w = fma(real(0.5), cs, real(0.5));
      dw = -(half_pi<real>() * sn);
    }
    sv = w * inv_r;
    dsv = (dw * P.inv_width - w * inv_r) * inv_r;
  } else {
    sv = real(0);
    dsv = real(0);
  }
}

// The environment's parameters checked on the host (DP_ERR_NULL / DP_ERR_TABLE_INFO).
inline int check_env(const dp_env_info *env) {
  if (!env) return set_error(DP_ERR_NULL, "env is NULL");
  if (!(env->rcs > 0.0) || !(env->rc > env->rcs))
    return set_error(DP_ERR_TABLE_INFO, "need 0 < rcs < rc (rcs %g, rc %g)", env->rcs, env->rc);
  if (env->kind != 0 && env->kind != 1) return set_error(DP_ERR_TABLE_INFO, "switch kind %d not 0 or 1", env->kind);
  if (!(env->std > 0.0) || !(env->std_all > 0.0))
    return set_error(DP_ERR_TABLE_INFO, "normalisation needs std > 0 and std_all > 0");
  if (!isfinite(env->mean)) return set_error(DP_ERR_TABLE_INFO, "normalisation mean not finite");
  return DP_OK;
}

}  // namespace
}  // namespace dpc
