// Fitting net (Sec. II: the descriptor D_i is passed to a fully connected
// network that outputs the atomic energy E_i; E = sum_i E_i) and its
// backward dE/dD_i, for the atoms of each centre type with that type's net.
//
// A hidden layer is a GEMM over the atoms of one type, [n x a] x [a x b],
// with the bias and tanh fused into its epilogue; the output layer (width 1)
// is a dot product per atom.  The backward runs the layers in reverse, one
// GEMM each against the transposed weights, with d tanh / dz = 1 - tanh^2
// applied as the operand is loaded and the skip term added in the epilogue.
//
// Only the tanh outputs of the hidden layers are kept (act, an output of the
// forward): a layer's input is the sum of the tanh outputs of its run of
// equal-width layers (the skips telescope: v_l = t_l + v_{l-1}), formed as
// the operand is loaded.
//
// GEMM tiling: small output tiles (FitTile below), 256 threads, 16-deep
// slices of both operands staged in shared memory.  Every FMA
// instruction has its 32 lanes busy; the kernels are bound by the FP64 pipe
// (f64) or the FP32 pipe (f32, df64).
#include <cuda_runtime.h>

#include <atomic>

#include "dp_common.cuh"

namespace dpc {
namespace {

// Output tile kBM x kBN per block, kTM x kTN per thread, 256 threads.
template <int BM, int BN, int TM, int TN>
struct Tile {
  static constexpr int kBM = BM, kBN = BN, kTM = TM, kTN = TN, kTX = BN / TN;  // kTX: threads across columns
  static_assert((BM / TM) * (BN / TN) == 256, "tile shape");
};
// By arithmetic and direction, measured on GB300 with the 240-wide nets of cu85 and water.  f64 is
// bound by the FP64 pipe alone, so its tiles are small: a type's few thousand atoms must still make
// many blocks per SM, or the SMs that get one block more than the others set the time (64 x 64
// tiles give 256 blocks for 4096 atoms on 152 SMs, 84 % at best; 16 x 16 tiles 3840, 97 %).  The
// backward's loader spends FP64 work on every element of A it stages (the factor 1 - t^2), once per
// column tile, so there wider tiles (16 x 48) pay for themselves.  df64 and f32 feed the FP32 pipes,
// where the shared-memory operand loads per product start to count: larger tiles.
template <typename real, bool kFwd>
struct FitTile {
  using T = Tile<16, 48, 1, 3>;
};
template <>
struct FitTile<double, true> {
  using T = Tile<16, 16, 1, 1>;
};
template <bool kFwd>
struct FitTile<float, kFwd> {
  using T = Tile<64, 64, 4, 4>;
};
template <>
struct FitTile<df64, true> {
  using T = Tile<32, 48, 2, 3>;
};
template <>
struct FitTile<df64, false> {
  using T = Tile<64, 64, 4, 4>;
};
constexpr int kBK = 16, kFitThreads = 256;
constexpr int kMaxChain = DP_MAX_LAYERS + 1;

__device__ __forceinline__ double tanh_r(const double z) { return tanh(z); }
__device__ __forceinline__ float tanh_r(const float z) { return tanhf(z); }
// df64: tanh in double on the FP64 pipe (one per output element, against a
// K-long df64 dot product per element on the FP32 pipes)
__device__ __forceinline__ df64 tanh_r(const df64 z) { return dfl::split(tanh(dfl::join(z))); }

template <typename real>
struct FitGemm {
  int64_t r0, n;  // the type's atoms: rows r0 .. r0 + n - 1
  int K, N;
  // forward operand: sum of nsrc row-major sources (D and/or tanh outputs), row strides lds
  const io_t<real> *src[kMaxChain];
  int64_t lds[kMaxChain];
  int nsrc;
  // backward operand: S (dE/dv, row stride ldS; NULL: S(i, o) = g_i wo[o]) times 1 - T^2
  const io_t<real> *S;
  int64_t ldS;
  const io_t<real> *g;   // [nloc] or NULL (= 1)
  const io_t<real> *wo;  // output-layer weights [K]
  const io_t<real> *T;
  int64_t ldT;
  const io_t<real> *W;     // forward: W [K][N]; backward: W [N][K] read as its transpose
  const io_t<real> *bias;  // forward: [N]
  bool skip;               // backward: add S(i, n) (the layer had an identity skip)
  io_t<real> *out;
  int64_t ldo;
};

template <typename real, bool kFwd>
__device__ __forceinline__ real load_a(const FitGemm<real> &P, int64_t row, int k) {
  if constexpr (kFwd) {
    io_t<real> v = P.src[0][row * P.lds[0] + k];
    for (int s = 1; s < P.nsrc; ++s) v += P.src[s][row * P.lds[s] + k];
    return from_io<real>(v);
  } else {
    const real t = from_io<real>(P.T[row * P.ldT + k]);
    real s;
    if (P.S)
      s = from_io<real>(P.S[row * P.ldS + k]);
    else
      s = from_io<real>(P.g ? P.g[row] : io_t<real>(1)) * from_io<real>(P.wo[k]);
    return s * fma(-t, t, real(1));
  }
}

template <typename real, bool kFwd>
__device__ __forceinline__ real load_b(const FitGemm<real> &P, int k, int nn) {
  if constexpr (kFwd)
    return from_io<real>(P.W[(size_t)k * P.N + nn]);
  else
    return from_io<real>(P.W[(size_t)nn * P.K + k]);
}

template <typename real, bool kFwd>
__global__ void __launch_bounds__(kFitThreads) fit_gemm_kernel(const FitGemm<real> P) {
  using TL = typename FitTile<real, kFwd>::T;
  constexpr int kBM = TL::kBM, kBN = TL::kBN, kTM = TL::kTM, kTN = TL::kTN, kTX = TL::kTX;
  __shared__ real As[kBK][kBM + 1];
  __shared__ real Bs[kBK][kBN];
  const int tx = threadIdx.x % kTX, ty = threadIdx.x / kTX;
  const int64_t m0 = (int64_t)blockIdx.y * kBM;
  const int n0 = blockIdx.x * kBN;
  real acc[kTM][kTN];
#pragma unroll
  for (int a = 0; a < kTM; ++a)
#pragma unroll
    for (int b = 0; b < kTN; ++b) acc[a][b] = real(0);
  for (int k0 = 0; k0 < P.K; k0 += kBK) {
    // A slice [kBM][kBK] and B slice [kBK][kBN], spread over the threads
    for (int e = threadIdx.x; e < kBM * kBK; e += kFitThreads) {
      const int am = e / kBK, ak = e - am * kBK;  // consecutive threads: consecutive k of one row
      const int64_t row = m0 + am;
      const int k = k0 + ak;
      As[ak][am] = (row < P.n && k < P.K) ? load_a<real, kFwd>(P, P.r0 + row, k) : real(0);
    }
    for (int e = threadIdx.x; e < kBK * kBN; e += kFitThreads) {
      const int bk = e / kBN, bn = e - bk * kBN;
      const int kb = k0 + bk, nb = n0 + bn;
      Bs[bk][bn] = (kb < P.K && nb < P.N) ? load_b<real, kFwd>(P, kb, nb) : real(0);
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kBK; ++kk) {
      real a[kTM], b[kTN];
#pragma unroll
      for (int q = 0; q < kTM; ++q) a[q] = As[kk][ty + (kBM / kTM) * q];
#pragma unroll
      for (int q = 0; q < kTN; ++q) b[q] = Bs[kk][tx + kTX * q];
#pragma unroll
      for (int p = 0; p < kTM; ++p)
#pragma unroll
        for (int q = 0; q < kTN; ++q) acc[p][q] = fma(a[p], b[q], acc[p][q]);
    }
    __syncthreads();
  }
  // epilogue: rows ty + (kBM / kTM) p, columns tx + kTX q (consecutive threads write consecutive columns)
#pragma unroll
  for (int p = 0; p < kTM; ++p) {
    const int64_t row = m0 + ty + (kBM / kTM) * p;
    if (row >= P.n) continue;
#pragma unroll
    for (int q = 0; q < kTN; ++q) {
      const int nn = n0 + tx + kTX * q;
      if (nn >= P.N) continue;
      real v = acc[p][q];
      if constexpr (kFwd) {
        v = tanh_r(v + from_io<real>(P.bias[nn]));
      } else if (P.skip) {
        const int64_t r = P.r0 + row;
        v += P.S ? from_io<real>(P.S[r * P.ldS + nn])
                 : from_io<real>(P.g ? P.g[r] : io_t<real>(1)) * from_io<real>(P.wo[nn]);
      }
      P.out[(P.r0 + row) * P.ldo + nn] = to_io(v);
    }
  }
}

// Output layer: E_i = v_{L-1} . wo + bo, one warp per atom, lanes over the inputs.
template <typename real>
__global__ void __launch_bounds__(128) fit_out_kernel(const FitGemm<real> P, const io_t<real> *bo, io_t<real> *E) {
  const int lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  if (i >= P.n) return;  // warp-uniform
  const int64_t row = P.r0 + i;
  real s = real(0);
  for (int k = lane; k < P.K; k += 32) s = fma(load_a<real, true>(P, row, k), from_io<real>(P.wo[k]), s);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += shfl_xor(s, o);
  if (lane == 0) E[row] = to_io(s + from_io<real>(bo[0]));
}

struct FitShape {
  int nlayer, ntypes;
  int w[DP_MAX_LAYERS + 1];
  int64_t P;       // parameters per type
  int64_t H;       // sum of hidden widths (row length of act)
  int maxh;        // largest hidden width
  int64_t woff[DP_MAX_LAYERS + 1];  // offset of W_l in a type's parameters (l >= 1)
  int64_t aoff[DP_MAX_LAYERS + 1];  // column offset of hidden layer l in act
  int64_t start[DP_MAX_TYPES + 1];
};

int fit_shape(const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start, FitShape *s) {
  if (!widths || !type_start) return set_error(DP_ERR_NULL, "widths or type_start is NULL");
  if (nlayer < 1 || nlayer > DP_MAX_LAYERS)
    return set_error(DP_ERR_UNSUPPORTED, "nlayer = %d outside [1, %d]", nlayer, DP_MAX_LAYERS);
  if (ntypes < 1 || ntypes > DP_MAX_TYPES)
    return set_error(DP_ERR_UNSUPPORTED, "ntypes = %d outside [1, %d]", ntypes, DP_MAX_TYPES);
  if (widths[nlayer] != 1) return set_error(DP_ERR_SHAPE, "the output layer has width %d, not 1", widths[nlayer]);
  s->nlayer = nlayer;
  s->ntypes = ntypes;
  s->P = 0;
  s->H = 0;
  s->maxh = 1;
  for (int l = 0; l <= nlayer; ++l) {
    if (widths[l] < 1 || widths[l] > (1 << 20)) return set_error(DP_ERR_SHAPE, "widths[%d] = %d", l, widths[l]);
    s->w[l] = widths[l];
  }
  for (int l = 1; l <= nlayer; ++l) {
    s->woff[l] = s->P;
    s->P += (int64_t)widths[l - 1] * widths[l] + widths[l];
    if (l < nlayer) {
      s->aoff[l] = s->H;
      s->H += widths[l];
      if (widths[l] > s->maxh) s->maxh = widths[l];
    }
  }
  for (int t = 0; t <= ntypes; ++t) {
    s->start[t] = type_start[t];
    if (t > 0 && type_start[t] < type_start[t - 1]) return set_error(DP_ERR_SHAPE, "type_start decreases");
  }
  if (type_start[0] != 0) return set_error(DP_ERR_SHAPE, "type_start[0] = %lld, not 0", (long long)type_start[0]);
  return DP_OK;
}

// Sources of the input of layer l (1 <= l <= nlayer): the tanh outputs of the run of
// equal-width layers that ends at l - 1, and D when that run reaches back to layer 0.
template <typename real>
void chain_sources(const FitShape &s, int l, const io_t<real> *D, const io_t<real> *act, FitGemm<real> &G) {
  G.nsrc = 0;
  int j = l - 1;
  while (true) {
    if (j == 0) {
      G.src[G.nsrc] = D;
      G.lds[G.nsrc++] = s.w[0];
      break;
    }
    G.src[G.nsrc] = act + s.aoff[j];
    G.lds[G.nsrc++] = s.H;
    if (s.w[j] != s.w[j - 1]) break;
    --j;
  }
}

template <typename real, bool kFwd>
int launch_gemm(const FitGemm<real> &G, cudaStream_t st, const char *who) {
  using TL = typename FitTile<real, kFwd>::T;
  const dim3 grid((unsigned)((G.N + TL::kBN - 1) / TL::kBN), (unsigned)((G.n + TL::kBM - 1) / TL::kBM));
  if (grid.y > 65535u) return set_error(DP_ERR_SHAPE, "%s: too many atoms of one type (%lld)", who, (long long)G.n);
  fit_gemm_kernel<real, kFwd><<<grid, kFitThreads, 0, st>>>(G);
  return launch_status(who);
}

template <typename real>
int fitting_fwd(const io_t<real> *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                const io_t<real> *D, io_t<real> *E, io_t<real> *act, void *stream) {
  clear_error();
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (!params || !D || !E || (s.H > 0 && !act)) return set_error(DP_ERR_NULL, "dp_fitting_fwd: NULL array");
  const cudaStream_t st = (cudaStream_t)stream;
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const io_t<real> *pt = params + (size_t)t * s.P;
    FitGemm<real> G{};
    G.r0 = s.start[t];
    G.n = n;
    for (int l = 1; l < nlayer; ++l) {  // hidden layers
      G.K = s.w[l - 1];
      G.N = s.w[l];
      chain_sources<real>(s, l, D, act, G);
      G.W = pt + s.woff[l];
      G.bias = G.W + (size_t)G.K * G.N;
      G.out = act + s.aoff[l];
      G.ldo = s.H;
      rc = launch_gemm<real, true>(G, st, "dp_fitting_fwd");
      if (rc) return rc;
    }
    G.K = s.w[nlayer - 1];
    G.N = 1;
    chain_sources<real>(s, nlayer, D, act, G);
    G.wo = pt + s.woff[nlayer];
    fit_out_kernel<real><<<(unsigned)((n + 3) / 4), 128, 0, st>>>(G, G.wo + G.K, E);
    rc = launch_status("dp_fitting_fwd");
    if (rc) return rc;
  }
  return DP_OK;
}

template <typename real>
int fitting_grad(const io_t<real> *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                 const io_t<real> *act, const io_t<real> *g, io_t<real> *dD, io_t<real> *work, void *stream) {
  clear_error();
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (!params || !dD || (s.H > 0 && !act) || (nlayer > 2 && !work))
    return set_error(DP_ERR_NULL, "dp_fitting_grad: NULL array");
  const cudaStream_t st = (cudaStream_t)stream;
  io_t<real> *buf[2] = {work, work ? work + (size_t)nloc * s.maxh : nullptr};
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const io_t<real> *pt = params + (size_t)t * s.P;
    FitGemm<real> G{};
    G.r0 = s.start[t];
    G.n = n;
    G.g = g;
    G.wo = pt + s.woff[nlayer];
    if (nlayer == 1) return set_error(DP_ERR_UNSUPPORTED, "a fitting net without hidden layers has dD = wo");
    const io_t<real> *S = nullptr;  // dE/dv of the layer being walked; NULL: g wo (the last hidden layer)
    int64_t ldS = 0;
    int cur = 0;
    for (int l = nlayer - 1; l >= 1; --l) {
      G.K = s.w[l];      // contraction over the layer's outputs
      G.N = s.w[l - 1];  // producing dE/dv_{l-1}
      G.S = S;
      G.ldS = ldS;
      G.T = act + s.aoff[l];
      G.ldT = s.H;
      G.W = pt + s.woff[l];
      G.skip = s.w[l] == s.w[l - 1];
      if (l == 1) {
        G.out = dD;
        G.ldo = s.w[0];
      } else {
        G.out = buf[cur];
        G.ldo = s.maxh;
      }
      rc = launch_gemm<real, false>(G, st, "dp_fitting_grad");
      if (rc) return rc;
      S = G.out;
      ldS = G.ldo;
      cur ^= 1;
    }
  }
  return DP_OK;
}

// ------------------------------------------------- backward without allocation
// Some callers cannot hand this library a scratch buffer: an MD engine's force
// loop that owns all device memory, sized once at start-up, and gives a plugin
// only its input and output arrays -- allocating there would synchronise the
// device in the middle of a time step and fragment the engine's pool.  For
// them dp_fitting_grad_noalloc_f64 takes its scratch (the two buffers the
// backward passes between layers) from this fixed array, which every GPU that
// loads the library keeps until the process exits.
constexpr size_t kStaticScratchDoubles = (size_t)1 << 20;  // 8 MiB
static __device__ __align__(256) double g_fit_scratch[kStaticScratchDoubles];

constexpr int kMaxScratchDevices = 64;
std::atomic<double *> g_fit_scratch_addr[kMaxScratchDevices];  // per device, filled on its first call

// Device address of the array on the current device.  In host code the array's
// name only stands in for it; the address comes from the runtime, looked up on
// the first call on each device and kept.
int static_scratch(double **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_fitting_grad_noalloc: cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxScratchDevices)
    return set_error(DP_ERR_UNSUPPORTED, "dp_fitting_grad_noalloc: device %d beyond the %d it tracks", dev,
                     kMaxScratchDevices);
  double *p = g_fit_scratch_addr[dev].load(std::memory_order_acquire);
  if (!p) {
    void *q = nullptr;
    e = cudaGetSymbolAddress(&q, g_fit_scratch);
    if (e != cudaSuccess)
      return set_error(DP_ERR_CUDA, "dp_fitting_grad_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    p = static_cast<double *>(q);
    g_fit_scratch_addr[dev].store(p, std::memory_order_release);
  }
  *out = p;
  return DP_OK;
}

int fitting_grad_noalloc(const double *params, const int32_t *widths, int nlayer, int ntypes,
                         const int64_t *type_start, const double *act, const double *g, double *dD, void *stream) {
  clear_error();
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  const size_t need = nlayer > 2 ? (size_t)2 * (size_t)nloc * (size_t)s.maxh : 0;
  if (need > kStaticScratchDoubles)
    return set_error(DP_ERR_UNSUPPORTED,
                     "dp_fitting_grad_noalloc: needs 2 x %lld atoms x %d = %zu doubles of scratch, the static array "
                     "holds %zu; use dp_fitting_grad_f64 with a work buffer",
                     (long long)nloc, s.maxh, need, kStaticScratchDoubles);
  double *work = nullptr;
  if (need > 0 && nloc > 0) {
    rc = static_scratch(&work);
    if (rc) return rc;
  }
  return fitting_grad<double>(params, widths, nlayer, ntypes, type_start, act, g, dD, work, stream);
}

}  // namespace
}  // namespace dpc

extern "C" {

int dp_fitting_grad_noalloc_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                                const int64_t *type_start, const double *act, const double *g, double *dD,
                                void *stream) {
  return dpc::fitting_grad_noalloc(params, widths, nlayer, ntypes, type_start, act, g, dD, stream);
}

int dp_fitting_fwd_f64(const double *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                       const double *D, double *E, double *act, void *stream) {
  return dpc::fitting_fwd<double>(params, widths, nlayer, ntypes, type_start, D, E, act, stream);
}
int dp_fitting_fwd_f32(const float *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                       const float *D, float *E, float *act, void *stream) {
  return dpc::fitting_fwd<float>(params, widths, nlayer, ntypes, type_start, D, E, act, stream);
}
int dp_fitting_fwd_df64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                        const int64_t *type_start, const double *D, double *E, double *act, void *stream) {
  return dpc::fitting_fwd<dpc::df64>(params, widths, nlayer, ntypes, type_start, D, E, act, stream);
}
int dp_fitting_grad_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                        const int64_t *type_start, const double *act, const double *g, double *dD, double *work,
                        void *stream) {
  return dpc::fitting_grad<double>(params, widths, nlayer, ntypes, type_start, act, g, dD, work, stream);
}
int dp_fitting_grad_f32(const float *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                        const float *act, const float *g, float *dD, float *work, void *stream) {
  return dpc::fitting_grad<float>(params, widths, nlayer, ntypes, type_start, act, g, dD, work, stream);
}
int dp_fitting_grad_df64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                         const int64_t *type_start, const double *act, const double *g, double *dD, double *work,
                         void *stream) {
  return dpc::fitting_grad<dpc::df64>(params, widths, nlayer, ntypes, type_start, act, g, dD, work, stream);
}

}  // extern "C"
