// Vector and tensor heads: the compressed path carried over to DP models of vectors and tensors
// (the paper's conclusion names both).  Up to T_i nothing changes; the head contracts the
// rotation-covariant rows k = 1..3 of T_i (the x, y, z columns of R~, Sec. II) with the M1
// rotation-invariant weights a_i a fitting net makes from D_i:
//   vector:  v_i[c]    = sum_m a_i[m] T_i[1+c][m]
//   tensor:  A_i[c][d] = sum_m a_i[m] (T_i[1+c][m] T_i[1+d][m])
// and their backward to dE/dT_i (added to the descriptor's, or overwriting) and dE/da_i.
//
// Forward: one warp per atom, lanes over the channels m (coalesced rows of T_i and a_i), the three
// (vector) or six (tensor: c <= d, mirrored) sums reduced across the warp in a fixed order.
// Backward: one thread per (atom, channel); dE/dv_i or dE/dA_i is read through L1 by the M1
// threads of the atom.  Both are bound by HBM (T_i, a_i and dT_i, da_i once each).
#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kHeadWarps = 4, kHeadThreads = 256;

template <typename real, bool kTensor>
__global__ void __launch_bounds__(kHeadWarps * 32)
    head_fwd_kernel(const real *__restrict__ T, const real *__restrict__ a, int64_t nloc, int M1,
                    real *__restrict__ out) {
  constexpr int kS = kTensor ? 6 : 3;  // tensor: (0,0) (0,1) (0,2) (1,1) (1,2) (2,2)
  const int lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * kHeadWarps + (threadIdx.x >> 5);
  if (i >= nloc) return;  // warp-uniform
  const real *Ti = T + i * 4 * M1, *ai = a + i * M1;
  real s[kS];
#pragma unroll
  for (int q = 0; q < kS; ++q) s[q] = real(0);
  for (int m = lane; m < M1; m += 32) {
    const real am = __ldg(ai + m);
    const real t0 = __ldg(Ti + M1 + m), t1 = __ldg(Ti + 2 * M1 + m), t2 = __ldg(Ti + 3 * M1 + m);
    if constexpr (kTensor) {
      s[0] = fma(am, t0 * t0, s[0]);
      s[1] = fma(am, t0 * t1, s[1]);
      s[2] = fma(am, t0 * t2, s[2]);
      s[3] = fma(am, t1 * t1, s[3]);
      s[4] = fma(am, t1 * t2, s[4]);
      s[5] = fma(am, t2 * t2, s[5]);
    } else {
      s[0] = fma(am, t0, s[0]);
      s[1] = fma(am, t1, s[1]);
      s[2] = fma(am, t2, s[2]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
#pragma unroll
    for (int q = 0; q < kS; ++q) s[q] += shfl_xor(s[q], o);
  if constexpr (kTensor) {
    if (lane < 9) {  // A[c][d] from the unique sum of {c, d}
      const int c = lane / 3, d = lane - 3 * (lane / 3);
      const int lo = c < d ? c : d, hi = c < d ? d : c;
      const int q = lo == 0 ? hi : lo == 1 ? 2 + hi : 5;
      real v = s[0];
#pragma unroll
      for (int r = 1; r < kS; ++r) v = q == r ? s[r] : v;
      out[i * 9 + lane] = v;
    }
  } else if (lane < 3) {
    out[i * 3 + lane] = lane == 0 ? s[0] : lane == 1 ? s[1] : s[2];
  }
}

template <typename real, bool kTensor>
__global__ void __launch_bounds__(kHeadThreads)
    head_grad_kernel(const real *__restrict__ T, const real *__restrict__ a, const real *__restrict__ dout,
                     int64_t nloc, int M1, real *__restrict__ dT, real *__restrict__ da, bool accumulate) {
  const int64_t e = (int64_t)blockIdx.x * kHeadThreads + threadIdx.x;
  if (e >= nloc * M1) return;
  const int64_t i = e / M1;
  const int m = (int)(e - i * M1);
  const real *Ti = T + i * 4 * M1;
  const real t[3] = {__ldg(Ti + M1 + m), __ldg(Ti + 2 * M1 + m), __ldg(Ti + 3 * M1 + m)};
  const real am = __ldg(a + e);
  real *dTi = dT ? dT + i * 4 * M1 : nullptr;
  real g[3], dam = real(0);
  if constexpr (kTensor) {
    const real *G = dout + i * 9;
    real Gm[9];
#pragma unroll
    for (int q = 0; q < 9; ++q) Gm[q] = __ldg(G + q);
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      real u = real(0);
#pragma unroll
      for (int d = 0; d < 3; ++d) {
        u = fma(Gm[3 * c + d] + Gm[3 * d + c], t[d], u);
        dam = fma(Gm[3 * c + d], t[c] * t[d], dam);
      }
      g[c] = am * u;
    }
  } else {
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      const real dv = __ldg(dout + i * 3 + c);
      g[c] = am * dv;
      dam = fma(dv, t[c], dam);
    }
  }
  if (!dT) {  // launch-uniform: only da wanted
  } else if (accumulate) {
#pragma unroll
    for (int c = 0; c < 3; ++c) dTi[(1 + c) * M1 + m] += g[c];
  } else {
    dTi[m] = real(0);
#pragma unroll
    for (int c = 0; c < 3; ++c) dTi[(1 + c) * M1 + m] = g[c];
  }
  if (da) da[e] = dam;
}

int head_check(const void *T, const void *a, const void *x, const void *y, int64_t nloc, int M1, const char *who) {
  if (nloc < 0) return set_error(DP_ERR_SHAPE, "%s: nloc = %lld", who, (long long)nloc);
  if (M1 < 1 || M1 > 4096) return set_error(DP_ERR_SHAPE, "%s: M1 = %d outside [1, 4096]", who, M1);
  if (nloc > 0 && (!T || !a || !x || !y)) return set_error(DP_ERR_NULL, "%s: NULL array", who);
  return DP_OK;
}

template <typename real, bool kTensor>
int head_fwd(const real *T, const real *a, int64_t nloc, int M1, real *out, void *stream, const char *who) {
  clear_error();
  int rc = head_check(T, a, out, out, nloc, M1, who);
  if (rc || nloc == 0) return rc;
  const int64_t blocks = (nloc + kHeadWarps - 1) / kHeadWarps;
  if (blocks > 0x7fffffffLL) return set_error(DP_ERR_SHAPE, "%s: nloc = %lld too large", who, (long long)nloc);
  head_fwd_kernel<real, kTensor><<<(unsigned)blocks, kHeadWarps * 32, 0, (cudaStream_t)stream>>>(T, a, nloc, M1, out);
  return launch_status(who);
}

template <typename real, bool kTensor>
int head_grad(const real *T, const real *a, const real *dout, int64_t nloc, int M1, real *dT, real *da,
              int accumulate, void *stream, const char *who) {
  clear_error();
  int rc = head_check(T, a, dout, dT ? (const void *)dT : (const void *)da, nloc, M1, who);
  if (rc || nloc == 0) return rc;
  const int64_t blocks = (nloc * M1 + kHeadThreads - 1) / kHeadThreads;
  if (blocks > 0x7fffffffLL) return set_error(DP_ERR_SHAPE, "%s: nloc = %lld too large", who, (long long)nloc);
  head_grad_kernel<real, kTensor><<<(unsigned)blocks, kHeadThreads, 0, (cudaStream_t)stream>>>(
      T, a, dout, nloc, M1, dT, da, accumulate != 0);
  return launch_status(who);
}

}  // namespace
}  // namespace dpc

extern "C" {

int dp_vector_head_f64(const double *T, const double *a, int64_t nloc, int M1, double *v, void *stream) {
  return dpc::head_fwd<double, false>(T, a, nloc, M1, v, stream, "dp_vector_head_f64");
}
int dp_vector_head_f32(const float *T, const float *a, int64_t nloc, int M1, float *v, void *stream) {
  return dpc::head_fwd<float, false>(T, a, nloc, M1, v, stream, "dp_vector_head_f32");
}
int dp_tensor_head_f64(const double *T, const double *a, int64_t nloc, int M1, double *A, void *stream) {
  return dpc::head_fwd<double, true>(T, a, nloc, M1, A, stream, "dp_tensor_head_f64");
}
int dp_tensor_head_f32(const float *T, const float *a, int64_t nloc, int M1, float *A, void *stream) {
  return dpc::head_fwd<float, true>(T, a, nloc, M1, A, stream, "dp_tensor_head_f32");
}
int dp_vector_head_grad_f64(const double *T, const double *a, const double *dv, int64_t nloc, int M1, double *dT,
                            double *da, int accumulate, void *stream) {
  return dpc::head_grad<double, false>(T, a, dv, nloc, M1, dT, da, accumulate, stream, "dp_vector_head_grad_f64");
}
int dp_vector_head_grad_f32(const float *T, const float *a, const float *dv, int64_t nloc, int M1, float *dT,
                            float *da, int accumulate, void *stream) {
  return dpc::head_grad<float, false>(T, a, dv, nloc, M1, dT, da, accumulate, stream, "dp_vector_head_grad_f32");
}
int dp_tensor_head_grad_f64(const double *T, const double *a, const double *dA, int64_t nloc, int M1, double *dT,
                            double *da, int accumulate, void *stream) {
  return dpc::head_grad<double, true>(T, a, dA, nloc, M1, dT, da, accumulate, stream, "dp_tensor_head_grad_f64");
}
int dp_tensor_head_grad_f32(const float *T, const float *a, const float *dA, int64_t nloc, int M1, float *dT,
                            float *da, int accumulate, void *stream) {
  return dpc::head_grad<float, true>(T, a, dA, nloc, M1, dT, da, accumulate, stream, "dp_tensor_head_grad_f32");
}

}  // extern "C"
