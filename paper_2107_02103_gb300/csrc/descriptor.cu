// Descriptor (Sec. II): S_i = T_i^T is M1 x 4, S_i^< its first M2 rows, and
// D_i = S_i (S_i^<)^T is M1 x M2:  D[i][m][n] = sum_k T[i][k][m] T[i][k][n].
//
// One warp per atom.  T_i (4 x M1) is staged in shared memory; the M1 x M2
// output tile is contiguous, so lane l computes elements l, l + 32, ... of it
// in storage order: every FP64 instruction has 32 busy lanes (M1*M2 is a
// multiple of 32 for the paper's shapes) and every store is coalesced.
// Both kernels also run in df64 arithmetic on double arrays (io_t).
#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kDescWarps = 4;

template <typename real>
__global__ void __launch_bounds__(kDescWarps * 32)
    descriptor_kernel(const io_t<real> *__restrict__ T, int64_t nloc, int M1, int M2, io_t<real> *__restrict__ D) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t i = (int64_t)blockIdx.x * kDescWarps + w;
  if (i >= nloc) return;  // warp-uniform; no block-wide barrier below
  real *Ts = reinterpret_cast<real *>(smem_raw) + (size_t)w * 4 * M1;
  const io_t<real> *__restrict__ Ti = T + i * 4 * M1;
#pragma unroll 4
  for (int e = lane; e < 4 * M1; e += 32) Ts[e] = from_io<real>(__ldg(Ti + e));
  __syncwarp();
  io_t<real> *__restrict__ Di = D + i * (int64_t)M1 * M2;
  const int total = M1 * M2;
  int m = lane / M2, n = lane - m * M2;
  const int dm = 32 / M2, dn = 32 - dm * M2;  // advance of (m, n) per 32 elements
  for (int e = lane; e < total; e += 32) {
    real v = Ts[m] * Ts[n];
    v = fma(Ts[M1 + m], Ts[M1 + n], v);
    v = fma(Ts[2 * M1 + m], Ts[2 * M1 + n], v);
    v = fma(Ts[3 * M1 + m], Ts[3 * M1 + n], v);
    Di[e] = to_io(v);
    m += dm;
    n += dn;
    if (n >= M2) {
      n -= M2;
      ++m;
    }
  }
}

// dD_i is staged in shared memory (read once, coalesced, converted once) in df64, where each
// element, read eight times, would otherwise cost eight conversions.  In f64 and f32 the
// second read of each element hits L1; staging there made the f32 kernel load-bound (both
// operands of every FMA from shared memory: 0.100 -> 0.146 ms on the water-like input).
template <typename real>
constexpr bool kStageDD = is_df64<real>;

// Shared memory per warp of the descriptor backward, in elements: T_i and the partial dT_i
// ([4][M1] each), and dD_i ([M1][M2 + 1], rows padded so that the eight rows one
// instruction reads fall in different banks) where it is staged.
template <typename real>
__host__ __device__ constexpr size_t desc_grad_smem_per_warp(int M1, int M2) {
  return (size_t)8 * M1 + (kStageDD<real> ? (size_t)M1 * (M2 + 1) : 0);
}

// Backward of the descriptor: D[m][n] = sum_k T[k][m] T[k][n] (n < M2) is
// quadratic in T, so for dD = dE/dD
//   dT[k][m] = sum_{n<M2} dD[m][n] T[k][n] + [m < M2] sum_{m'} dD[m'][m] T[k][m'].
// One warp per atom.  The 4*M1 (m, k) pairs of the first term are spread
// over the lanes (lane l: pairs l, l + 32, ...; 8 rows x 4 k per step, so the
// dD row reads of a step are 8 rows of M2 values); the 4*M2 (k, m) pairs of
// the second term walk the M1 rows of dD, each step reading one row.  Both
// terms meet in shared memory and dT is written coalesced.
template <typename real>
__global__ void __launch_bounds__(kDescWarps * 32)
    descriptor_grad_kernel(const io_t<real> *__restrict__ T, const io_t<real> *__restrict__ dD, int64_t nloc, int M1,
                           int M2, io_t<real> *__restrict__ dT) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t i = (int64_t)blockIdx.x * kDescWarps + w;
  if (i >= nloc) return;  // warp-uniform; no block-wide barrier below
  real *Ts = reinterpret_cast<real *>(smem_raw) + (size_t)w * desc_grad_smem_per_warp<real>(M1, M2);  // [4][M1]
  real *Gs = Ts + 4 * M1;                                                                              // [4][M1]
  const io_t<real> *__restrict__ Ti = T + i * 4 * M1;
  const io_t<real> *__restrict__ Di = dD + i * (int64_t)M1 * M2;
#pragma unroll 4
  for (int e = lane; e < 4 * M1; e += 32) Ts[e] = from_io<real>(__ldg(Ti + e));
  // dD_i into shared memory ([M1][M2] after Gs) where staged; every element is read 8 times
  const real *Ds = Gs + 4 * M1;
  if constexpr (kStageDD<real>) {
    real *Dw = Gs + 4 * M1;
    // unrolled so that each lane has eight loads in flight, not one
#pragma unroll 8
    for (int e = lane; e < M1 * M2; e += 32) {
      const int r = e / M2;
      Dw[e + r] = from_io<real>(__ldg(Di + e));
    }
  }
  __syncwarp();
  auto dd = [&](int m, int n) -> real {  // dD_i[m][n]
    if constexpr (kStageDD<real>) return Ds[m * (M2 + 1) + n];
    else return __ldg(Di + (size_t)m * M2 + n);
  };
  // In df64 each sum runs in four interleaved partial sums: one chain of dependent df64 FMAs
  // (eight dependent instructions each) would leave the pipes idle between them.  In f64 and
  // f32 the extra adds cost more than they hide (f64: +13 % on the water-like input).
  constexpr int NP = is_df64<real> ? 4 : 1;
  // first term, pairs p = 4 m + k
  for (int p = lane; p < 4 * M1; p += 32) {
    const int m = p >> 2, k = p & 3;
    const real *tk = Ts + k * M1;
    real v[NP];
#pragma unroll
    for (int q = 0; q < NP; ++q) v[q] = real(0);
    int n = 0;
    for (; n + NP <= M2; n += NP)
#pragma unroll
      for (int q = 0; q < NP; ++q) v[q] = fma(dd(m, n + q), tk[n + q], v[q]);
    for (; n < M2; ++n) v[0] = fma(dd(m, n), tk[n], v[0]);
#pragma unroll
    for (int q = 1; q < NP; ++q) v[0] += v[q];
    Gs[k * M1 + m] = v[0];
  }
  __syncwarp();
  // second term, pairs p = M2 k + m (m < M2)
  for (int p = lane; p < 4 * M2; p += 32) {
    const int k = p / M2, m = p - k * M2;
    const real *tk = Ts + k * M1;
    real v[NP];
#pragma unroll
    for (int q = 0; q < NP; ++q) v[q] = real(0);
    int mp = 0;
    for (; mp + NP <= M1; mp += NP)
#pragma unroll
      for (int q = 0; q < NP; ++q) v[q] = fma(dd(mp + q, m), tk[mp + q], v[q]);
    for (; mp < M1; ++mp) v[0] = fma(dd(mp, m), tk[mp], v[0]);
#pragma unroll
    for (int q = 1; q < NP; ++q) v[0] += v[q];
    Gs[k * M1 + m] += v[0];
  }
  __syncwarp();
  io_t<real> *__restrict__ dTi = dT + i * 4 * M1;
  for (int e = lane; e < 4 * M1; e += 32) dTi[e] = to_io(Gs[e]);
}

template <typename real>
int descriptor_grad(const io_t<real> *T, const io_t<real> *dD, int64_t nloc, int M1, int M2, io_t<real> *dT,
                    void *stream) {
  clear_error();
  if (nloc < 0 || M1 < 1 || M2 < 1 || M2 > M1)
    return set_error(DP_ERR_SHAPE, "need nloc >= 0 and 1 <= M2 <= M1 (nloc %lld, M1 %d, M2 %d)", (long long)nloc, M1,
                     M2);
  if (M1 > 4096) return set_error(DP_ERR_UNSUPPORTED, "M1 = %d > 4096", M1);
  if (nloc == 0) return DP_OK;
  if (!T || !dD || !dT) return set_error(DP_ERR_NULL, "T, dD or dT is NULL");
  const int64_t blocks = (nloc + kDescWarps - 1) / kDescWarps;
  if (blocks > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
  const size_t smem = (size_t)kDescWarps * desc_grad_smem_per_warp<real>(M1, M2) * sizeof(real);
  if (smem > 227 * 1024) return set_error(DP_ERR_UNSUPPORTED, "M1 = %d, M2 = %d need too much shared memory", M1, M2);
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(descriptor_grad_kernel<real>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_descriptor_contract_grad: %s", cudaGetErrorString(e));
  }
  descriptor_grad_kernel<real>
      <<<(unsigned)blocks, kDescWarps * 32, smem, (cudaStream_t)stream>>>(T, dD, nloc, M1, M2, dT);
  return launch_status("dp_descriptor_contract_grad");
}

template <typename real>
int descriptor(const io_t<real> *T, int64_t nloc, int M1, int M2, io_t<real> *D, void *stream) {
  clear_error();
  if (nloc < 0 || M1 < 1 || M2 < 1 || M2 > M1)
    return set_error(DP_ERR_SHAPE, "need nloc >= 0 and 1 <= M2 <= M1 (nloc %lld, M1 %d, M2 %d)", (long long)nloc, M1,
                     M2);
  if (M1 > 4096) return set_error(DP_ERR_UNSUPPORTED, "M1 = %d > 4096", M1);
  if (nloc == 0) return DP_OK;
  if (!T || !D) return set_error(DP_ERR_NULL, "T or D is NULL");
  const int64_t blocks = (nloc + kDescWarps - 1) / kDescWarps;
  if (blocks > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
  const size_t smem = (size_t)kDescWarps * 4 * M1 * sizeof(real);
  if (smem > 227 * 1024) return set_error(DP_ERR_UNSUPPORTED, "M1 = %d needs too much shared memory", M1);
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(descriptor_kernel<real>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)smem);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_descriptor_contract: %s", cudaGetErrorString(e));
  }
  descriptor_kernel<real><<<(unsigned)blocks, kDescWarps * 32, smem, (cudaStream_t)stream>>>(T, nloc, M1, M2, D);
  return launch_status("dp_descriptor_contract");
}

}  // namespace

}  // namespace dpc

extern "C" {

int dp_descriptor_contract_f64(const double *T, int64_t nloc, int M1, int M2, double *D, void *stream) {
  return dpc::descriptor<double>(T, nloc, M1, M2, D, stream);
}

int dp_descriptor_contract_f32(const float *T, int64_t nloc, int M1, int M2, float *D, void *stream) {
  return dpc::descriptor<float>(T, nloc, M1, M2, D, stream);
}

int dp_descriptor_contract_df64(const double *T, int64_t nloc, int M1, int M2, double *D, void *stream) {
  return dpc::descriptor<dpc::df64>(T, nloc, M1, M2, D, stream);
}

int dp_descriptor_contract_grad_df64(const double *T, const double *dD, int64_t nloc, int M1, int M2, double *dT,
                                     void *stream) {
  return dpc::descriptor_grad<dpc::df64>(T, dD, nloc, M1, M2, dT, stream);
}

int dp_descriptor_contract_grad_f64(const double *T, const double *dD, int64_t nloc, int M1, int M2, double *dT,
                                    void *stream) {
  return dpc::descriptor_grad<double>(T, dD, nloc, M1, M2, dT, stream);
}

int dp_descriptor_contract_grad_f32(const float *T, const float *dD, int64_t nloc, int M1, int M2, float *dT,
                                    void *stream) {
  return dpc::descriptor_grad<float>(T, dD, nloc, M1, M2, dT, stream);
}

}  // extern "C"
