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

#include <algorithm>
#include <atomic>
#include <cstdint>

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

// ------------------------------------------------- f64 GEMMs on the tensor cores
// GB300 retires FP64 at 2 lanes per clock per SM, fp16 products on the tensor
// cores (mma.sync, measured) at about 480 times that rate.  An f64 GEMM
// C = A B is recovered from fp16 products by splitting every operand element
// into base-32 digits (the error-free splitting of Ozaki et al.):
//   a_ik = 2^E_i sum_{s=1..11} A_s[i][k] 32^-s + r_ik,  A_s integers in [-31, 31],  |r_ik| < 2^(E_i - 55),
// with max_k |a_ik| < 2^E_i, and likewise b_kj with a column exponent F_j, so that
//   C_ij = 2^(E_i + F_j) sum_{d=2..12} 32^-d sum_{s+t=d} (A_s B_t)_ij + (terms with s + t > 12 and the r).
// Every (A_s B_t)_ij is a sum of integer products |A_s B_t| <= 961, so its fp32
// sum on the tensor cores is exact while it stays below 2^24: the 11 diagonals
// d are summed in fp32 over at most kFlushK = 1024 of K at a time (11 pairs x
// 1024 x 961 < 2^24) and then added into an f64 accumulator.  What rounds is
// that f64 accumulation (11 adds per 1024 of K), the 55-bit truncation of the
// operands and the dropped terms: |error| <~ K 2^-51 max_k|a_ik| max_k|b_kj|,
// against K 2^-53 sum_k |a_ik b_kj| for an f64 dot product.  A row or column
// with an inf or NaN gives NaN outputs.
//
// Block tile 32 x 80 (ten warps of 16 x 16), 32-deep K slices: per slice the
// block's A rows are split into 11 fp16 digit planes in shared memory (their
// exponents found by a pass over the rows first), the pre-split B planes are
// copied in, and each warp runs the 66 digit products of its tile as
// m16n8k16 MMAs with fp32 accumulators, one per diagonal.
namespace tc {
constexpr int kS = 11;  // digits per operand element
constexpr int kBM = 32, kBN = 80, kBK = 32;
constexpr int kLd = kBK + 8;  // shared row stride in halves (80 B): the 8 rows an ldmatrix reads hit 8 distinct bank groups
constexpr int kWarpsN = kBN / 16, kWarps = (kBM / 16) * kWarpsN, kThreads = 32 * kWarps;
constexpr int kFlushK = 1024;
constexpr int kNonFinite = 1 << 20;  // exponent of a row or column holding inf or NaN
constexpr size_t kSmemA = (size_t)kS * kBM * kLd * 2, kSmemB = (size_t)kS * kBN * kLd * 2;
constexpr size_t kSmem = kSmemA + kSmemB + (size_t)(kBM + kBN) * sizeof(int);
static_assert((size_t)kS * kFlushK * 961 < (1u << 24), "fp32 diagonal sums must stay exact");
static_assert((kS * kBN * (kBK / 8)) % kThreads == 0, "B copy: whole rounds");

__host__ __device__ constexpr int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

__device__ __forceinline__ int exp_bits(double x) { return (int)(((uint64_t)__double_as_longlong(x) >> 52) & 0x7ff); }
// E with max |x| < 2^E from the largest biased exponent (normal x: |x| < 2^(eb - 1022))
__device__ __forceinline__ int exp_of_max(int ebmax) { return ebmax == 0x7ff ? kNonFinite : max(ebmax, 1) - 1022; }

// |x| 2^-E as an integer with 55 fractional bits, truncated; below 2^55 since |x| < 2^E
__device__ __forceinline__ uint64_t fixed55(double x, int E) {
  const uint64_t b = (uint64_t)__double_as_longlong(x);
  const int eb = (int)((b >> 52) & 0x7ff);
  const uint64_t mant = b & 0xfffffffffffffull;
  const uint64_t m = eb ? (mant | (1ull << 52)) : mant;
  const int sh = (eb ? eb - 1075 : -1074) - E + 55;  // |x| 2^(55 - E) = m 2^sh, sh <= 2 for finite x
  if (sh >= 0) return m << min(sh, 10);
  return sh > -64 ? m >> -sh : 0ull;
}

// The kS digits of two fixed-point values, digit s of both packed as an fp16 pair (element 0 in the
// low half), each with its element's sign: 0x6400 | d is the fp16 1024 + d, and 1024 comes off exactly.
__device__ __forceinline__ void digit_pairs(uint64_t f0, uint64_t f1, uint32_t sign2, uint32_t (&h)[kS]) {
#pragma unroll
  for (int s = 1; s <= kS; ++s) {
    const uint32_t d0 = (uint32_t)(f0 >> (55 - 5 * s)) & 31u, d1 = (uint32_t)(f1 >> (55 - 5 * s)) & 31u;
    uint32_t v;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(v) : "r"(0x64006400u | d0 | (d1 << 16)), "r"(0x64006400u));
    h[s - 1] = v ^ sign2;
  }
}

__device__ __forceinline__ uint32_t sign_pair(double x0, double x1) {
  return (uint32_t)((uint64_t)__double_as_longlong(x0) >> 63) << 15 | (uint32_t)((uint64_t)__double_as_longlong(x1) >> 63)
                                                                          << 31;
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

__device__ __forceinline__ void mma_f16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
               : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
               : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src));
}

// B of one layer as digit planes [kS][Np][Kp] (fp16, column n's K values contiguous) and the column
// exponents F [Np]; columns >= N and rows >= K are zero.  Forward: B[k][n] = W[k][n] (W is [K][N]);
// backward: B[k][n] = W[n][k].  One warp per column.
__global__ void __launch_bounds__(128) split_b_kernel(const double *__restrict__ W, int K, int N, bool fwd, int Np,
                                                      int Kp, uint32_t *__restrict__ planes, int *__restrict__ Fexp) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * 4 + (threadIdx.x >> 5);
  if (n >= Np) return;  // warp-uniform
  auto w = [&](int k) {
    return (n < N && k < K) ? (fwd ? W[(size_t)k * N + n] : W[(size_t)n * K + k]) : 0.0;
  };
  int eb = 0;
  for (int k = lane; k < K; k += 32) eb = max(eb, exp_bits(w(k)));
  const int F = exp_of_max(__reduce_max_sync(0xffffffffu, eb));
  if (lane == 0) Fexp[n] = F;
  for (int c2 = lane; c2 < Kp / 2; c2 += 32) {
    const double x0 = w(2 * c2), x1 = w(2 * c2 + 1);
    uint32_t h[kS];
    digit_pairs(fixed55(x0, F), fixed55(x1, F), sign_pair(x0, x1), h);
#pragma unroll
    for (int s = 0; s < kS; ++s) planes[((size_t)s * Np + n) * (Kp / 2) + c2] = h[s];
  }
}

template <bool kFwd>
__global__ void __launch_bounds__(kThreads) gemm_kernel(const FitGemm<double> P, const uint16_t *__restrict__ planes,
                                                        const int *__restrict__ Fexp, int Np, int Kp) {
  extern __shared__ __align__(16) unsigned char smem[];
  uint16_t *As = reinterpret_cast<uint16_t *>(smem);           // [kS][kBM][kLd]
  uint16_t *Bs = reinterpret_cast<uint16_t *>(smem + kSmemA);  // [kS][kBN][kLd]
  int *sE = reinterpret_cast<int *>(smem + kSmemA + kSmemB);   // row exponents [kBM]
  int *sF = sE + kBM;                                          // column exponents [kBN]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int wm = warp / kWarpsN, wn = warp - wm * kWarpsN;
  const int64_t m0 = (int64_t)blockIdx.y * kBM;
  const int n0 = blockIdx.x * kBN;

  // row exponents of the block's rows over the whole of K, and the columns' exponents
  for (int r = warp; r < kBM; r += kWarps) {
    const int64_t row = m0 + r;
    int eb = 0;
    if (row < P.n)
      for (int k = lane; k < P.K; k += 32) eb = max(eb, exp_bits(load_a<double, kFwd>(P, P.r0 + row, k)));
    eb = __reduce_max_sync(0xffffffffu, eb);
    if (lane == 0) sE[r] = exp_of_max(eb);
  }
  for (int c = threadIdx.x; c < kBN; c += kThreads) sF[c] = Fexp[n0 + c];
  __syncthreads();

  float acc[kS][2][4];
#pragma unroll
  for (int d = 0; d < kS; ++d)
#pragma unroll
    for (int j = 0; j < 2; ++j)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[d][j][c] = 0.f;
  double acc64[2][4];
#pragma unroll
  for (int j = 0; j < 2; ++j)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc64[j][c] = 0.0;

  int since_flush = 0;
  for (int k0 = 0; k0 < P.K; k0 += kBK) {  // uniform
    // B planes: kS x kBN rows of kBK halves, 16 B per copy
#pragma unroll 1
    for (int e = threadIdx.x; e < kS * kBN * (kBK / 8); e += kThreads) {
      const int s = e / (kBN * (kBK / 8)), rem = e - s * kBN * (kBK / 8);
      const int nn = rem / (kBK / 8), kc = rem - nn * (kBK / 8);
      cp_async16(smem_u32(Bs + (s * kBN + nn) * kLd + kc * 8),
                 planes + ((size_t)s * Np + n0 + nn) * Kp + k0 + kc * 8);
    }
    asm volatile("cp.async.commit_group;");
    // A: the block's rows split into digit planes, two adjacent columns per thread
    uint32_t *As32 = reinterpret_cast<uint32_t *>(As);
#pragma unroll 1
    for (int e = threadIdx.x; e < kBM * kBK / 2; e += kThreads) {
      const int r = e / (kBK / 2), c2 = e - r * (kBK / 2);
      const int64_t row = m0 + r;
      const int k = k0 + 2 * c2;
      double x0 = 0.0, x1 = 0.0;
      if (row < P.n) {
        if (k < P.K) x0 = load_a<double, kFwd>(P, P.r0 + row, k);
        if (k + 1 < P.K) x1 = load_a<double, kFwd>(P, P.r0 + row, k + 1);
      }
      const int E = sE[r];
      uint32_t h[kS];
      digit_pairs(fixed55(x0, E), fixed55(x1, E), sign_pair(x0, x1), h);
#pragma unroll
      for (int s = 0; s < kS; ++s) As32[(s * kBM + r) * (kLd / 2) + c2] = h[s];
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
#pragma unroll
    for (int ks = 0; ks < kBK / 16; ++ks) {
      uint32_t a[kS][4];
#pragma unroll
      for (int s = 0; s < kS; ++s)
        ldmatrix_x4(a[s], smem_u32(As + (s * kBM + wm * 16 + (lane & 15)) * kLd + ks * 16 + (lane >> 4) * 8));
#pragma unroll
      for (int t = 0; t < kS; ++t) {
        uint32_t b[4];
        ldmatrix_x4(b, smem_u32(Bs + (t * kBN + wn * 16 + (lane & 7) + ((lane >> 4) << 3)) * kLd + ks * 16 +
                                ((lane >> 3) & 1) * 8));
#pragma unroll
        for (int s = 0; s + t < kS; ++s) {  // digits s + 1 and t + 1: diagonal s + t + 2 <= kS + 1
          mma_f16(acc[s + t][0], a[s], b[0], b[1]);
          mma_f16(acc[s + t][1], a[s], b[2], b[3]);
        }
      }
    }
    __syncthreads();
    since_flush += kBK;
    if (since_flush == kFlushK || k0 + kBK >= P.K) {  // uniform: the diagonals into f64, smallest first
      since_flush = 0;
#pragma unroll
      for (int d = kS - 1; d >= 0; --d) {
        const double scale = __hiloint2double((1023 - 5 * (d + 2)) << 20, 0);  // 32^-(d + 2)
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            acc64[j][c] = fma(dfl::widen(acc[d][j][c]), scale, acc64[j][c]);
            acc[d][j][c] = 0.f;
          }
      }
    }
  }

  // epilogue: lane (gid, tig) holds rows gid and gid + 8, columns 2 tig and 2 tig + 1 of each 8-wide tile
  const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
  for (int j = 0; j < 2; ++j)
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int rl = wm * 16 + gid + (c >= 2 ? 8 : 0), cl = wn * 16 + j * 8 + 2 * tig + (c & 1);
      const int64_t row = m0 + rl;
      const int nn = n0 + cl;
      if (row >= P.n || nn >= P.N) continue;
      const int E = sE[rl], F = sF[cl];
      double v = (E >= kNonFinite || F >= kNonFinite) ? __longlong_as_double(0x7ff8000000000000ll)
                                                     : scalbn(acc64[j][c], E + F);
      if constexpr (kFwd) {
        v = tanh(v + P.bias[nn]);
      } else if (P.skip) {
        const int64_t r = P.r0 + row;
        v += P.S ? P.S[r * P.ldS + nn] : (P.g ? P.g[r] : 1.0) * P.wo[nn];
      }
      P.out[(P.r0 + row) * P.ldo + nn] = v;
    }
}

// Where the B planes and column exponents of each hidden-layer GEMM of one type sit in the work
// buffer (forward: layers 1 .. L-1; backward: L-1 .. 1), and the bytes they take.
struct Layer {
  int K, N, Np, Kp;
  size_t planes, fexp;  // byte offsets
};
size_t layout(const FitShape &s, bool fwd, Layer *out) {
  size_t off = 0;
  for (int q = 0; q + 1 < s.nlayer; ++q) {
    const int l = fwd ? q + 1 : s.nlayer - 1 - q;
    Layer &L = out[q];
    L.K = fwd ? s.w[l - 1] : s.w[l];
    L.N = fwd ? s.w[l] : s.w[l - 1];
    L.Np = (int)round_up(L.N, kBN);
    L.Kp = (int)round_up(L.K, kBK);
    L.planes = off;
    off += (size_t)round_up((int64_t)kS * L.Np * L.Kp * 2, 256);
    L.fexp = off;
    off += (size_t)round_up((int64_t)L.Np * 4, 256);
  }
  return off;
}

size_t work_bytes(const FitShape &s, int64_t nloc) {
  Layer L[DP_MAX_LAYERS];
  size_t b = std::max(layout(s, true, L), layout(s, false, L));
  if (s.nlayer > 2) b += (size_t)2 * (size_t)nloc * (size_t)s.maxh * sizeof(double);
  return b;
}

int set_smem() {
  static std::atomic<bool> done{false};
  if (done.load(std::memory_order_acquire)) return DP_OK;
  for (auto k : {&gemm_kernel<true>, &gemm_kernel<false>}) {
    const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_fitting_*_tc_f64: %s", cudaGetErrorString(e));
  }
  done.store(true, std::memory_order_release);
  return DP_OK;
}

int split(const double *W, const Layer &L, bool fwd, unsigned char *work, cudaStream_t st, const char *who) {
  split_b_kernel<<<(unsigned)((L.Np + 3) / 4), 128, 0, st>>>(W, L.K, L.N, fwd, L.Np, L.Kp,
                                                            reinterpret_cast<uint32_t *>(work + L.planes),
                                                            reinterpret_cast<int *>(work + L.fexp));
  return launch_status(who);
}

template <bool kFwd>
int gemm(const FitGemm<double> &G, const Layer &L, const unsigned char *work, cudaStream_t st, const char *who) {
  const dim3 grid((unsigned)(L.Np / kBN), (unsigned)((G.n + kBM - 1) / kBM));
  if (grid.y > 65535u) return set_error(DP_ERR_SHAPE, "%s: too many atoms of one type (%lld)", who, (long long)G.n);
  gemm_kernel<kFwd><<<grid, kThreads, kSmem, st>>>(G, reinterpret_cast<const uint16_t *>(work + L.planes),
                                                   reinterpret_cast<const int *>(work + L.fexp), L.Np, L.Kp);
  return launch_status(who);
}

int check_work(const FitShape &s, int64_t nloc, const void *work, size_t nbytes, const char *who) {
  const size_t need = work_bytes(s, nloc);
  if (need > 0 && !work) return set_error(DP_ERR_NULL, "%s: work is NULL", who);
  if (nbytes < need) return set_error(DP_ERR_SHAPE, "%s: work holds %zu bytes, needs %zu", who, nbytes, need);
  if (reinterpret_cast<uintptr_t>(work) % 256) return set_error(DP_ERR_SHAPE, "%s: work is not 256-byte aligned", who);
  return DP_OK;
}

int fwd(const double *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start, const double *D,
        double *E, double *act, void *work, size_t work_nbytes, void *stream) {
  clear_error();
  static const char *who = "dp_fitting_fwd_tc_f64";
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (!params || !D || !E || (s.H > 0 && !act)) return set_error(DP_ERR_NULL, "%s: NULL array", who);
  if ((rc = check_work(s, nloc, work, work_nbytes, who)) || (rc = set_smem())) return rc;
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(work);
  Layer L[DP_MAX_LAYERS];
  layout(s, true, L);
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const double *pt = params + (size_t)t * s.P;
    for (int l = 1; l < nlayer; ++l)  // this type's weights as digit planes (the previous type's are done with)
      if ((rc = split(pt + s.woff[l], L[l - 1], true, wk, st, who))) return rc;
    FitGemm<double> G{};
    G.r0 = s.start[t];
    G.n = n;
    for (int l = 1; l < nlayer; ++l) {
      G.K = s.w[l - 1];
      G.N = s.w[l];
      chain_sources<double>(s, l, D, act, G);
      G.W = pt + s.woff[l];
      G.bias = G.W + (size_t)G.K * G.N;
      G.out = act + s.aoff[l];
      G.ldo = s.H;
      if ((rc = gemm<true>(G, L[l - 1], wk, st, who))) return rc;
    }
    G.K = s.w[nlayer - 1];
    G.N = 1;
    chain_sources<double>(s, nlayer, D, act, G);
    G.wo = pt + s.woff[nlayer];
    fit_out_kernel<double><<<(unsigned)((n + 3) / 4), 128, 0, st>>>(G, G.wo + G.K, E);
    if ((rc = launch_status(who))) return rc;
  }
  return DP_OK;
}

int grad(const double *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
         const double *act, const double *g, double *dD, void *work, size_t work_nbytes, void *stream) {
  clear_error();
  static const char *who = "dp_fitting_grad_tc_f64";
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (nlayer == 1) return set_error(DP_ERR_UNSUPPORTED, "a fitting net without hidden layers has dD = wo");
  if (!params || !dD || (s.H > 0 && !act)) return set_error(DP_ERR_NULL, "%s: NULL array", who);
  if ((rc = check_work(s, nloc, work, work_nbytes, who)) || (rc = set_smem())) return rc;
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(work);
  Layer L[DP_MAX_LAYERS];
  Layer Lf[DP_MAX_LAYERS];
  const size_t planes = std::max(layout(s, true, Lf), layout(s, false, L));
  double *buf[2] = {reinterpret_cast<double *>(wk + planes),
                    reinterpret_cast<double *>(wk + planes) + (size_t)nloc * s.maxh};
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const double *pt = params + (size_t)t * s.P;
    for (int q = 0; q + 1 < nlayer; ++q)
      if ((rc = split(pt + s.woff[nlayer - 1 - q], L[q], false, wk, st, who))) return rc;
    FitGemm<double> G{};
    G.r0 = s.start[t];
    G.n = n;
    G.g = g;
    G.wo = pt + s.woff[nlayer];
    const double *S = nullptr;
    int64_t ldS = 0;
    int cur = 0;
    for (int l = nlayer - 1; l >= 1; --l) {
      G.K = s.w[l];
      G.N = s.w[l - 1];
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
      if ((rc = gemm<false>(G, L[nlayer - 1 - l], wk, st, who))) return rc;
      S = G.out;
      ldS = G.ldo;
      cur ^= 1;
    }
  }
  return DP_OK;
}

size_t work_bytes_api(const int32_t *widths, int nlayer, int64_t nloc) {
  clear_error();
  if (nloc < 0) return 0;
  const int64_t ts[2] = {0, nloc};
  FitShape s{};
  if (fit_shape(widths, nlayer, 1, ts, &s)) return 0;
  return work_bytes(s, nloc);
}
}  // namespace tc

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

size_t dp_fitting_tc_work_bytes(const int32_t *widths, int nlayer, int64_t nloc) {
  return dpc::tc::work_bytes_api(widths, nlayer, nloc);
}
int dp_fitting_fwd_tc_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                          const int64_t *type_start, const double *D, double *E, double *act, void *work,
                          size_t work_bytes, void *stream) {
  return dpc::tc::fwd(params, widths, nlayer, ntypes, type_start, D, E, act, work, work_bytes, stream);
}
int dp_fitting_grad_tc_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                           const int64_t *type_start, const double *act, const double *g, double *dD, void *work,
                           size_t work_bytes, void *stream) {
  return dpc::tc::grad(params, widths, nlayer, ntypes, type_start, act, g, dD, work, work_bytes, stream);
}

}  // extern "C"
