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

// f64 and df64: tanh evaluated in double-float on the FP32 pipes (dfl::tanh_d), not on the FP64
// pipe, where a double tanh costs about a tenth of a 240-deep layer's products
__device__ __forceinline__ double tanh_r(const double z) { return dfl::tanh_d(z); }
__device__ __forceinline__ float tanh_r(const float z) { return tanhf(z); }
__device__ __forceinline__ df64 tanh_r(const df64 z) { return dfl::split(dfl::tanh_d(dfl::join(z))); }

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
// GB300 retires FP64 at 2 lanes per clock per SM but fp16 products on its
// tcgen05 tensor cores at ~1000 times that rate.  An f64 GEMM C = A B is
// recovered from fp16 products by splitting every operand element into base-64
// digits (the error-free splitting of Ozaki et al.):
//   a_ik = 2^E_i sum_{s=1..9} A_s[i][k] 64^-s + r_ik,  A_s integers in [-63, 63],  |r_ik| < 2^(E_i - 54),
// with max_k |a_ik| < 2^E_i, and likewise b_kj with a column exponent F_j, so that
//   C_ij = 2^(E_i + F_j) sum_{d=2..10} 64^-d sum_{s+t=d} (A_s B_t)_ij + (terms with s + t > 10 and the r).
// Every (A_s B_t)_ij is a sum of integer products |A_s B_t| <= 3969; a diagonal
// d has at most 9 of them, so its fp32 sum on the tensor cores is exact while
// a block's share of K is at most kMaxShareK = 448 (9 x 448 x 3969 < 2^24).
// The 9 diagonal sums of an output are combined on the FP32 pipe into four
// floats (the two largest by an exact two-sum, the rest in float-float, whose
// rounding lies ~2^-60 below the result); epilogue_kernel adds the shares'
// floats into a three-float sum by exact two-sums and converts it to f64 once.
// What rounds is that conversion, the 54-bit truncation of the operands and
// the dropped terms: |error| <~ K 2^-50 max_k|a_ik| max_k|b_kj|, against
// K 2^-53 sum_k |a_ik b_kj| for an f64 dot product.  A row or column with an
// inf or NaN gives NaN outputs.
//
// gemm_kernel: one CTA of 128 threads per 128 x 48 output tile and share of K,
// one CTA per SM (its 9 diagonal accumulators take 432 of the SM's 512 TMEM
// columns).  The digit planes of A (per chunk of rows) and B (per call) are
// made by split_rows_kernel, once per element, as the shared-memory image of
// each (tile, 16-deep K slice) block: the tcgen05 K-major layout without
// swizzle (8-row x 16-byte core matrices).  Lane 0 of warp 0 moves a slice's
// A and B blocks into one of four stages with two bulk async copies counted in
// bytes on the stage's "full" mbarrier; lane 0 of warp 1 issues the slice's 45
// digit-product MMAs (M 128, N 48, K 16, fp16 in, fp32 accumulators in TMEM,
// one per diagonal) and commits them to the stage's "empty" mbarrier, which
// the producer waits on before refilling the stage.  A last commit on a
// barrier used once releases the four warps, which read their TMEM lane
// quadrant (rows), combine the diagonals and write the share's result as four
// floats; epilogue_kernel sums the shares in a fixed order, scales by 2^(E+F)
// and applies the layer's epilogue.  A is always a plain matrix: the forward
// keeps each layer's input v_l (tanh outputs plus the skip) in a work buffer,
// the backward writes dE/dv (for the next skip) and dE/dv (1 - t^2) (the next
// A).  Every wait on an mbarrier is bounded; a wait that gives up makes the
// tile's outputs NaN.
namespace tc {
constexpr int kS = 9;      // digits per operand element
constexpr int kBits = 6;   // bits per digit
constexpr int kFrac = kS * kBits;  // 54 fractional bits
constexpr int kTM = 128, kTN = 48, kTK = 16;  // CTA tile; K per stage (one MMA)
constexpr int kStages = 4;
constexpr int kThreads = 128;  // one warp per TMEM lane quadrant; lane 0 of warps 0 and 1: producer and MMA issuer
constexpr int kMaxShareK = 448;
constexpr int kNonFinite = 1 << 20;  // exponent of a row or column holding inf or NaN
constexpr uint32_t kLBO = 128, kSBO = 256;  // core matrices: next along K at +128 B, next 8 rows at +256 B
constexpr int kPlaneA = kTM * kTK * 2, kPlaneB = kTN * kTK * 2;  // bytes of one digit plane in a stage
constexpr int kStageBytes = kS * (kPlaneA + kPlaneB);
constexpr uint32_t kTmemCols = 512;  // allocation (a power of two); kS * kTN = 432 used
constexpr size_t kSmemTotal = (size_t)kStages * kStageBytes + (2 * kStages + 1) * 8 + 16;
static_assert((size_t)kS * kMaxShareK * 63 * 63 < (1u << 24), "fp32 diagonal sums must stay exact");
static_assert(kMaxShareK % kTK == 0 && kS * kTN <= (int)kTmemCols, "shares and TMEM");
static_assert(kSmemTotal <= 227 * 1024, "shared memory per block");

__host__ __device__ constexpr int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

__device__ __forceinline__ int exp_bits(double x) { return (int)(((uint64_t)__double_as_longlong(x) >> 52) & 0x7ff); }
// E with max |x| < 2^E from the largest biased exponent (normal x: |x| < 2^(eb - 1022))
__device__ __forceinline__ int exp_of_max(int ebmax) { return ebmax == 0x7ff ? kNonFinite : max(ebmax, 1) - 1022; }

// |x| 2^-E as an integer with kFrac fractional bits, truncated; below 2^kFrac since |x| < 2^E
__device__ __forceinline__ uint64_t fixed_point(double x, int E) {
  const uint64_t b = (uint64_t)__double_as_longlong(x);
  const int eb = (int)((b >> 52) & 0x7ff);
  const uint64_t mant = b & 0xfffffffffffffull;
  const uint64_t m = eb ? (mant | (1ull << 52)) : mant;
  const int sh = (eb ? eb - 1075 : -1074) - E + kFrac;  // |x| 2^(kFrac - E) = m 2^sh, sh <= 1 for finite x
  if (sh >= 0) return m << min(sh, 10);
  return sh > -64 ? m >> -sh : 0ull;
}

// The kS digits of two fixed-point values, digit s of both packed as an fp16 pair (element 0 in the
// low half), each with its element's sign: 0x6400 | d is the fp16 1024 + d, and 1024 comes off exactly.
__device__ __forceinline__ void digit_pairs(uint64_t f0, uint64_t f1, uint32_t sign2, uint32_t (&h)[kS]) {
  constexpr uint32_t kMask = (1u << kBits) - 1;
#pragma unroll
  for (int s = 1; s <= kS; ++s) {
    const uint32_t d0 = (uint32_t)(f0 >> (kFrac - kBits * s)) & kMask;
    const uint32_t d1 = (uint32_t)(f1 >> (kFrac - kBits * s)) & kMask;
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

// Rows of a matrix as digit planes, laid out as the shared-memory image of each (tile of RT rows,
// 16-deep K slice) block that gemm_kernel copies in one piece: block (r / RT, k / 16) holds the kS
// planes of those rows and columns, plane s at s RT 32 bytes, and in a plane the tcgen05 K-major
// core matrices (8 rows x 8 k = 128 bytes; the second 8 k of the slice at +128 B, the next 8 rows
// at +256 B).  Also the rows' exponents [rows_p].  Element (r, k) of the source is X[r ld_r + k ld_k];
// rows >= nrows and columns >= K are zero (row_exps_kernel first finds the exponents).  Used for the A operand (rows of the
// layer input, RT = kTM) and for B (RT = kTN; forward: the columns of W, ld_r = 1, ld_k = N;
// backward: the rows of W).
__global__ void __launch_bounds__(128) row_exps_kernel(const double *__restrict__ X, int64_t ld_r, int64_t ld_k,
                                                       int64_t nrows, int K, int64_t rows_p, int *__restrict__ exps) {
  // one warp per row: E with max_k |x_rk| < 2^E
  const int lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  if (r >= rows_p) return;  // warp-uniform
  int eb = 0;
  if (r < nrows)
    for (int k = lane; k < K; k += 32) eb = max(eb, exp_bits(__ldg(X + r * ld_r + k * ld_k)));
  eb = __reduce_max_sync(0xffffffffu, eb);
  if (lane == 0) exps[r] = exp_of_max(eb);
}

constexpr int kSplitK = 64;  // K per warp of split_rows_kernel
__global__ void __launch_bounds__(128) split_rows_kernel(const double *__restrict__ X, int64_t ld_r, int64_t ld_k,
                                                         int64_t nrows, int K, int64_t rows_p, int Kp, int RT,
                                                         unsigned char *__restrict__ planes,
                                                         const int *__restrict__ exps) {
  // one warp per (group of 8 rows, kSplitK of K): lane = (row ri8 = lane / 4, pair of k kp = lane % 4),
  // so that per plane and 8 k the warp writes one whole 128-byte core matrix
  const int lane = threadIdx.x & 31, ri8 = lane >> 2, kp = lane & 3;
  const int kchunks = (Kp + kSplitK - 1) / kSplitK;
  const int64_t w = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  const int64_t g = w / kchunks;  // 8-row group
  if (g * 8 >= rows_p) return;    // warp-uniform
  const int kc = (int)(w - g * kchunks);
  const int64_t r = g * 8 + ri8;
  const double *__restrict__ xr = X + (r < nrows ? r : 0) * ld_r;
  auto x = [&](int k) { return (r < nrows && k < K) ? __ldg(xr + k * ld_k) : 0.0; };
  const int E = exps[r];
  const size_t plane = (size_t)RT * kTK * 2, block = kS * plane;
  const int ri = (int)(r % RT);
  unsigned char *rowbase = planes + (size_t)(r / RT) * (Kp / kTK) * block + (ri >> 3) * kSBO + (ri & 7) * 16 + kp * 4;
  for (int k0 = kc * kSplitK; k0 < min(Kp, kc * kSplitK + kSplitK); k0 += 8) {
    const int k = k0 + 2 * kp;
    const double x0 = x(k), x1 = x(k + 1);
    uint32_t h[kS];
    digit_pairs(fixed_point(x0, E), fixed_point(x1, E), sign_pair(x0, x1), h);
    unsigned char *dst = rowbase + (size_t)(k0 / kTK) * block + ((k0 % kTK) >> 3) * kLBO;
#pragma unroll
    for (int s = 0; s < kS; ++s) *reinterpret_cast<uint32_t *>(dst + s * plane) = h[s];
  }
}

// One hidden-layer GEMM of a chunk of one type's atoms: rows r0 .. r0 + n - 1 of the plain
// row-major A [*][K] (as digit planes) times B (digit planes), K cut into shares of at most
// kMaxShareK (grid z); the shares' f64 results go to `part`, and epilogue_kernel sums them and
// applies the layer's epilogue.
struct TcGemm {
  int64_t r0, n;  // output rows r0 .. r0 + n - 1; A's planes hold rows 0 .. n - 1 of this chunk
  int K, N;
  const double *A;  // the layer input itself (forward: its skip term)
  int64_t lda;
  const unsigned char *aplanes;  // A's blocks [Mp / kTM][Kp / kTK] of kS x kPlaneA bytes
  const int *Eexp;          // [Mp]
  int64_t Mp;
  const unsigned char *planes;   // B's blocks [Np / kTN][Kp / kTK] of kS x kPlaneB bytes
  const int *Fexp;
  int Np, Kp;
  float4 *part;             // [ksplit][Mp][Np]: each share's result (grid z) as four floats, see gemm_kernel
  int slices_per_split;
  bool skip;
  // forward
  const double *bias;
  double *act;
  int64_t ldact;
  double *V;
  int64_t ldv;
  // backward
  const double *S;  // NULL: S(row, col) = g_row wo_col
  int64_t ldS;
  const double *g, *wo;
  const double *T;  // tanh outputs of the layer below (NULL: the last GEMM)
  int64_t ldT;
  double *Snext, *Z;
  int64_t ldz;
  double *out;
  int64_t ldo;
};

// shared-memory descriptor of a K-major operand without swizzle (tcgen05): start address, the byte
// offsets of the next core matrix along K (leading) and along the rows (stride), version 1
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFF) >> 4) | ((uint64_t)(kLBO >> 4) << 16) | ((uint64_t)(kSBO >> 4) << 32) |
         (1ull << 46);
}
// instruction descriptor, kind::f16: D f32 (bits 4-5 = 1), A and B f16 (0), both K-major, N >> 3 at
// bit 17 (set per MMA), M >> 4 at bit 24
constexpr uint32_t kIdescNoN = (1u << 4) | ((uint32_t)(kTM >> 4) << 24);  // N >> 3 goes in at bit 17
constexpr int kMaxPlanesPerMma = 256 / kTN;  // N <= 256 for M = 128
static_assert(kTN % 16 == 0 && kMaxPlanesPerMma >= 1, "MMA N: multiples of 16 up to 256");

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  uint32_t done = 0;
  for (int it = 0; it < (1 << 24) && !done; ++it)
    asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
                 : "=r"(done)
                 : "r"(bar), "r"(parity)
                 : "memory");
  return done != 0;
}

__global__ void __launch_bounds__(kThreads, 1) gemm_kernel(const TcGemm P) {
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + kStages * kStageBytes);  // stage loaded
  uint64_t *empty = full + kStages;                                               // stage's MMAs done
  uint64_t *done = empty + kStages;                                               // every MMA done (one use)
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(done + 1);
  int *flags = reinterpret_cast<int *>(tmem_holder + 1);                          // producer / issuer ok
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t m0 = (int64_t)blockIdx.y * kTM;
  const int n0 = blockIdx.x * kTN;
  const int nslices = P.Kp / kTK;
  const int i0 = blockIdx.z * P.slices_per_split;
  const int nsl = min(nslices - i0, P.slices_per_split);  // > 0: no empty share

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(full + s)));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(empty + s)));
    }
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(done)));
    asm volatile("fence.mbarrier_init.release.cluster;");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  const uint32_t tmem = *tmem_holder;
  const uint32_t sbase = smem_u32(smem);
  bool ok = true;

  if (warp == 0 && lane == 0) {
    // producer: each slice's A and B blocks, one bulk copy each, counted in bytes on the stage's
    // "full" barrier; a stage is reused once the MMAs that read it have completed ("empty")
    const unsigned char *asrc = P.aplanes + ((size_t)blockIdx.y * nslices + i0) * (kS * kPlaneA);
    const unsigned char *bsrc = P.planes + ((size_t)blockIdx.x * nslices + i0) * (kS * kPlaneB);
    for (int j = 0; j < nsl && ok; ++j) {
      const int st = j % kStages;
      if (j >= kStages) ok = mbar_wait(smem_u32(empty + st), (uint32_t)((j / kStages - 1) & 1));
      if (!ok) break;
      const uint32_t bar = smem_u32(full + st), dst = sbase + st * kStageBytes;
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"((uint32_t)kStageBytes)
                   : "memory");
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                   "l"(asrc + (size_t)j * (kS * kPlaneA)), "r"((uint32_t)(kS * kPlaneA)), "r"(bar)
                   : "memory");
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                       dst + kS * kPlaneA),
                   "l"(bsrc + (size_t)j * (kS * kPlaneB)), "r"((uint32_t)(kS * kPlaneB)), "r"(bar)
                   : "memory");
    }
  } else if (warp == 1 && lane == 0) {
    // MMA issuer: the 45 digit products of each slice once it has landed, then a commit that frees the stage
    for (int i = 0; i < nsl && ok; ++i) {
      const int st = i % kStages;
      ok = mbar_wait(smem_u32(full + st), (uint32_t)((i / kStages) & 1));
      if (!ok) break;
      asm volatile("tcgen05.fence::after_thread_sync;");
      const uint64_t a0 = smem_desc(sbase + st * kStageBytes), b0 = smem_desc(sbase + st * kStageBytes + kS * kPlaneA);
      // Digit s of A against digits t = 0 .. kS-1-s of B in one MMA: B's planes lie back to back in
      // the stage (48 rows each, one row stride), so together they are one operand of 48 (kS - s)
      // rows, and with the accumulator address moved by s diagonals the block of plane t lands on
      // diagonal s + t.  N is at most 256, so up to 5 planes (240 columns) per MMA: 13 MMAs per
      // slice instead of 45, each reading its A tile once for up to 240 columns.
#pragma unroll
      for (int s = 0; s < kS; ++s) {
        const uint64_t ad = a0 + (uint64_t)((s * kPlaneA) >> 4);  // start-address field, in 16-byte units
#pragma unroll
        for (int t0 = 0; t0 < kS - s; t0 += kMaxPlanesPerMma) {
          const int np = min(kMaxPlanesPerMma, kS - s - t0);
          const uint64_t bd = b0 + (uint64_t)((t0 * kPlaneB) >> 4);
          const uint32_t idesc = kIdescNoN | ((uint32_t)((np * kTN) >> 3) << 17);
          const uint32_t acc = (i > 0 || s > 0) ? 1u : 0u;  // digit 1 of A writes every diagonal first
          asm volatile(
              "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
              " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem + (uint32_t)((s + t0) * kTN)),
              "l"(ad), "l"(bd), "r"(idesc), "r"(acc));
        }
      }
      asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(empty + st)));
    }
    // one more commit, on a barrier used once: it completes when every MMA issued above has (also
    // after a wait that gave up, so that nobody waits on it in vain)
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(done)));
  }
  if (lane == 0 && warp < 2) flags[warp] = ok;
  __syncwarp();
  // The other warps wait here rather than on a stage barrier: a parity wait can only tell apart the
  // current phase and the one before, and they would start it phases ahead of the MMAs.
  __syncthreads();
  ok = flags[0] && flags[1];
  ok = mbar_wait(smem_u32(done), 0) && ok;
  asm volatile("tcgen05.fence::after_thread_sync;");

  // combine the diagonals of row 32 (warp % 4) + lane (the warp's TMEM lane quadrant), the warp's
  // third of the columns, 8 at a time
  const int rl = 32 * (warp & 3) + lane;
  float4 *outp = P.part + ((size_t)blockIdx.z * P.Mp + m0 + rl) * P.Np + n0;
  const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
  constexpr int kColsPerWarp = kTN / (kThreads / 128);
  static_assert(kColsPerWarp % 8 == 0, "column share");
#pragma unroll 1
  for (int c0 = (warp >> 2) * kColsPerWarp; c0 < (warp >> 2) * kColsPerWarp + kColsPerWarp; c0 += 8) {
    float v[kS][8];
#pragma unroll
    for (int d = 0; d < kS; ++d)
      asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                   : "=f"(v[d][0]), "=f"(v[d][1]), "=f"(v[d][2]), "=f"(v[d][3]), "=f"(v[d][4]), "=f"(v[d][5]),
                     "=f"(v[d][6]), "=f"(v[d][7])
                   : "r"(trow + (uint32_t)(d * kTN + c0)));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      // sum_d v_d 64^-(d+2) as four floats on the FP32 pipe: diagonals 2 and 3 (d = 0, 1) as an exact
      // two-sum, 4 .. 10 in float-float, smallest first (its rounding lies ~2^-60 below the sum).
      // The scaling by 2^(E+F), and all f64 arithmetic, is left to epilogue_kernel.
      dfl::df64 lo(0.0f);
#pragma unroll
      for (int d = kS - 1; d >= 2; --d) {
        const float x = v[d][c] * __uint_as_float((uint32_t)(127 - kBits * (d + 2)) << 23);  // exact: 64^-(d+2)
        lo = lo + dfl::df64(x);
      }
      const float a = v[0][c] * 0x1p-12f, b = v[1][c] * 0x1p-18f;  // exact
      const float s = __fadd_rn(a, b), bb = __fsub_rn(s, a);
      const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
      outp[c0 + c] = ok ? make_float4(s, e, lo.hi, lo.lo) : make_float4(__int_as_float(0x7fc00000), 0.f, 0.f, 0.f);
    }
  }

  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

// The layer's epilogue over the chunk's n x N outputs, from the shares' partial results summed in
// a fixed order (so a call's results do not depend on timing):
//   forward:  t = tanh(acc + bias); act[row][col] = t; V[row][col] = t (+ A[row][col] when the layer
//             keeps its width: the identity skip, v_l = t_l + v_{l-1})
//   backward: s = acc (+ S[row][col] or g_row wo_col when the layer kept its width); then either
//             out[row][col] = s (dE/dD, the last GEMM) or S_next[row][col] = s and
//             Z[row][col] = s (1 - t_prev^2) with t_prev = T[row][col] (the next GEMM's A)
// f 2^e as a double, exactly, by moving fields (f finite; |e| < 900, so a normal result stays normal
// and a float that is zero stays zero; float subnormals, which the sums do not produce, widen to 0)
__device__ __forceinline__ double widen_pow2(float f, int e) {
  const double d = dfl::widen(f);
  const long long b = __double_as_longlong(d);
  return (b & 0x7fffffffffffffffll) ? __longlong_as_double(b + ((long long)e << 52)) : d;
}

template <bool kFwd>
__global__ void __launch_bounds__(256) epilogue_kernel(const TcGemm P, int ksplit) {
  // rows over the grid, columns over the block (no 64-bit division per element)
  for (int64_t rc = blockIdx.x; rc < P.n; rc += gridDim.x)
  for (int nn = threadIdx.x; nn < P.N; nn += blockDim.x) {
    const int64_t row = P.r0 + rc;
    // the shares' four floats each, added into a three-float sum by exact two-sums on the FP32 pipe
    // (only the last component rounds, ~2^-72 below the sum), then one conversion to f64 and the
    // scaling by the row and column powers of two
    float s0 = 0.f, s1 = 0.f, s2 = 0.f;
    auto add = [&](float x) {
      float t = __fadd_rn(s0, x), z = __fsub_rn(t, s0);
      const float e0 = __fadd_rn(__fsub_rn(s0, __fsub_rn(t, z)), __fsub_rn(x, z));
      s0 = t;
      t = __fadd_rn(s1, e0);
      z = __fsub_rn(t, s1);
      const float e1 = __fadd_rn(__fsub_rn(s1, __fsub_rn(t, z)), __fsub_rn(e0, z));
      s1 = t;
      s2 = __fadd_rn(s2, e1);
    };
    for (int z = 0; z < ksplit; ++z) {
      const float4 q = P.part[((size_t)z * P.Mp + rc) * P.Np + nn];
      add(q.x);
      add(q.y);
      add(q.z);
      add(q.w);
    }
    const int E = P.Eexp[rc], F = P.Fexp[nn];
    double v;
    if (E >= kNonFinite || F >= kNonFinite || s0 != s0)
      v = __longlong_as_double(0x7ff8000000000000ll);
    else if (E + F > -900 && E + F < 900)  // the scaling moves exponent fields only (sums stay normal)
      v = __dadd_rn(__dadd_rn(widen_pow2(s0, E + F), widen_pow2(s1, E + F)), widen_pow2(s2, E + F));
    else
      v = scalbn(__dadd_rn(__dadd_rn(dfl::widen(s0), dfl::widen(s1)), dfl::widen(s2)), E + F);
    if constexpr (kFwd) {
      const double t = dfl::tanh_d(v + P.bias[nn]);
      P.act[row * P.ldact + nn] = t;
      P.V[row * P.ldv + nn] = P.skip ? t + P.A[row * P.lda + nn] : t;
    } else {
      if (P.skip) v += P.S ? P.S[row * P.ldS + nn] : (P.g ? P.g[row] : 1.0) * P.wo[nn];
      if (P.T) {
        const double t = P.T[row * P.ldT + nn];
        P.Snext[row * P.ldz + nn] = v;
        P.Z[row * P.ldz + nn] = v * fma(-t, t, 1.0);
      } else {
        P.out[row * P.ldo + nn] = v;
      }
    }
  }
}

// dz of the last hidden layer: Z[row][k] = g_row wo_k (1 - t_k^2), t its tanh outputs
__global__ void __launch_bounds__(256) last_dz_kernel(int64_t r0, int64_t n, int K, const double *__restrict__ g,
                                                      const double *__restrict__ wo, const double *__restrict__ T,
                                                      int64_t ldT, double *__restrict__ Z, int64_t ldz) {
  for (int64_t rr = blockIdx.x; rr < n; rr += gridDim.x)
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int64_t row = r0 + rr;
    const double t = T[row * ldT + k];
    Z[row * ldz + k] = (g ? g[row] : 1.0) * wo[k] * fma(-t, t, 1.0);
  }
}

// Where the B planes and column exponents of each hidden-layer GEMM of one type sit in the work
// buffer (forward: layers 1 .. L-1; backward: L-1 .. 1).  After them come the A planes and row
// exponents of one chunk of at most kChunkRows atoms, and the [nloc][max hidden width] buffers
// between layers (forward: 2, backward: 4).
constexpr int64_t kChunkRows = 16384;
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
    L.Np = (int)round_up(L.N, kTN);
    L.Kp = (int)round_up(L.K, kTK);
    L.planes = off;
    off += (size_t)round_up((int64_t)kS * L.Np * L.Kp * 2, 256);
    L.fexp = off;
    off += (size_t)round_up((int64_t)L.Np * 4, 256);
  }
  return off;
}

struct WorkMap {
  size_t bplanes;          // bytes of the B planes (the larger of the two directions)
  size_t aplanes, aexp;    // byte offsets of the A planes and row exponents of one chunk
  int64_t Mp;              // rows of A planes per chunk
  int Kpmax;
  size_t part;             // byte offset of the shares' partial results
  size_t buffers;          // byte offset of the buffers between layers
};

// K shares of one GEMM: at most kMaxShareK each (the exactness bound), and more when the tiles
// alone would not give every SM a few CTAs (one CTA per SM), but at least kMinShareSlices slices
// each (a CTA's pipeline fill and combine are paid once per share).
constexpr int kMaxShareSlices = kMaxShareK / kTK;
constexpr int64_t kTargetCtas = 4 * 152;
constexpr int kMinShareSlices = 6;
int ksplit_for(int64_t Mp, int Np, int Kp) {
  const int64_t tiles = (Mp / kTM) * (Np / kTN);
  const int slices = Kp / kTK;
  int want = (int)std::min<int64_t>((kTargetCtas + tiles - 1) / tiles, std::max(1, slices / kMinShareSlices));
  want = std::max(want, (slices + kMaxShareSlices - 1) / kMaxShareSlices);
  const int per = (slices + want - 1) / want;
  return (slices + per - 1) / per;  // no empty share; per <= kMaxShareSlices
}

WorkMap work_map(const FitShape &s, int64_t nloc) {
  Layer L[DP_MAX_LAYERS];
  WorkMap m{};
  m.bplanes = std::max(layout(s, true, L), layout(s, false, L));
  int kmax = 1;
  for (int l = 0; l < s.nlayer; ++l) kmax = std::max(kmax, s.w[l]);  // every GEMM's K is a layer width
  m.Kpmax = (int)round_up(kmax, kTK);
  int64_t maxn = 0;  // rows of the largest type
  for (int t = 0; t < s.ntypes; ++t) maxn = std::max<int64_t>(maxn, s.start[t + 1] - s.start[t]);
  m.Mp = round_up(std::min<int64_t>(std::max<int64_t>(maxn, 1), kChunkRows), kTM);
  m.aplanes = m.bplanes;
  m.aexp = m.aplanes + (size_t)round_up((int64_t)kS * m.Mp * m.Kpmax * 2, 256);
  m.part = m.aexp + (size_t)round_up(m.Mp * 4, 256);
  // shares x Mp x Np over the GEMMs: below kTargetCtas tiles plus the largest chunk's Mp x Np, or
  // the exactness bound's shares at the largest chunk (a smaller chunk stays under both)
  int Npmax = kTN;
  for (int l = 0; l < s.nlayer; ++l) Npmax = std::max(Npmax, (int)round_up(s.w[l], kTN));
  int64_t part = kTargetCtas * kTM * kTN + m.Mp * Npmax;
  for (int q = 0; q + 1 < s.nlayer; ++q)
    for (int dir = 0; dir < 2; ++dir) {
      layout(s, dir == 0, L);
      part = std::max<int64_t>(part, (int64_t)ksplit_for(m.Mp, L[q].Np, L[q].Kp) * m.Mp * L[q].Np);
    }
  m.buffers = m.part + (size_t)round_up(part * 16, 256);
  return m;
}

size_t work_bytes(const FitShape &s, int64_t nloc) {
  const WorkMap m = work_map(s, nloc);
  return m.buffers + (s.nlayer > 1 ? (size_t)4 * (size_t)nloc * (size_t)s.maxh * sizeof(double) : 0);
}

int set_smem() {
  static std::atomic<bool> done{false};
  if (done.load(std::memory_order_acquire)) return DP_OK;
  const cudaError_t e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemTotal);
  if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_fitting_*_tc_f64: %s", cudaGetErrorString(e));
  done.store(true, std::memory_order_release);
  return DP_OK;
}

int split_rows(const double *X, int64_t ld_r, int64_t ld_k, int64_t nrows, int K, int64_t rows_p, int Kp, int RT,
               unsigned char *planes, unsigned char *exps, cudaStream_t st, const char *who) {
  row_exps_kernel<<<(unsigned)((rows_p + 3) / 4), 128, 0, st>>>(X, ld_r, ld_k, nrows, K, rows_p,
                                                                 reinterpret_cast<int *>(exps));
  int rc = launch_status(who);
  if (rc) return rc;
  const int64_t warps = rows_p / 8 * ((Kp + kSplitK - 1) / kSplitK);
  split_rows_kernel<<<(unsigned)((warps + 3) / 4), 128, 0, st>>>(X, ld_r, ld_k, nrows, K, rows_p, Kp, RT, planes,
                                                                 reinterpret_cast<const int *>(exps));
  return launch_status(who);
}

// The weights of one layer as B planes: forward B[k][n] = W[k][n] (W is [K][N]), backward B[k][n] = W[n][k]
int split_b(const double *W, const Layer &L, bool fwd, unsigned char *work, cudaStream_t st, const char *who) {
  return fwd ? split_rows(W, 1, L.N, L.N, L.K, L.Np, L.Kp, kTN, work + L.planes, work + L.fexp, st, who)
             : split_rows(W, L.K, 1, L.N, L.K, L.Np, L.Kp, kTN, work + L.planes, work + L.fexp, st, who);
}

// G over its rows in chunks of at most kChunkRows: each chunk's A rows split into planes, then the GEMM
template <bool kFwd>
int gemm(TcGemm G, const Layer &L, unsigned char *work, const WorkMap &m, cudaStream_t st, const char *who) {
  G.planes = work + L.planes;
  G.Fexp = reinterpret_cast<const int *>(work + L.fexp);
  G.Np = L.Np;
  G.Kp = L.Kp;
  G.aplanes = work + m.aplanes;
  G.Eexp = reinterpret_cast<const int *>(work + m.aexp);
  G.part = reinterpret_cast<float4 *>(work + m.part);
  const int64_t r_end = G.r0 + G.n;
  for (int64_t r0 = G.r0; r0 < r_end; r0 += kChunkRows) {
    TcGemm C = G;
    C.r0 = r0;
    C.n = std::min<int64_t>(kChunkRows, r_end - r0);
    C.Mp = round_up(C.n, kTM);
    int rc = split_rows(G.A + r0 * G.lda, G.lda, 1, C.n, G.K, C.Mp, L.Kp, kTM, work + m.aplanes, work + m.aexp, st, who);
    if (rc) return rc;
    const int ksplit = ksplit_for(C.Mp, L.Np, L.Kp);
    C.slices_per_split = (L.Kp / kTK + ksplit - 1) / ksplit;
    const dim3 grid((unsigned)(L.Np / kTN), (unsigned)(C.Mp / kTM), (unsigned)ksplit);
    gemm_kernel<<<grid, kThreads, kSmemTotal, st>>>(C);
    if ((rc = launch_status(who))) return rc;
    epilogue_kernel<kFwd><<<(unsigned)std::min<int64_t>(C.n, 152 * 32), 256, 0, st>>>(C, ksplit);
    if ((rc = launch_status(who))) return rc;
  }
  return DP_OK;
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
  const WorkMap m = work_map(s, nloc);
  double *V[2] = {reinterpret_cast<double *>(wk + m.buffers), nullptr};
  V[1] = V[0] + (size_t)nloc * s.maxh;
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const double *pt = params + (size_t)t * s.P;
    for (int l = 1; l < nlayer; ++l)  // this type's weights as digit planes (the previous type's are done with)
      if ((rc = split_b(pt + s.woff[l], L[l - 1], true, wk, st, who))) return rc;
    const double *in = D;  // v_{l-1}: D, then the layer outputs with their skips
    int64_t ldin = s.w[0];
    for (int l = 1; l < nlayer; ++l) {
      TcGemm G{};
      G.r0 = s.start[t];
      G.n = n;
      G.K = s.w[l - 1];
      G.N = s.w[l];
      G.A = in;
      G.lda = ldin;
      G.skip = s.w[l] == s.w[l - 1];
      G.bias = pt + s.woff[l] + (size_t)G.K * G.N;
      G.act = act + s.aoff[l];
      G.ldact = s.H;
      G.V = V[(l - 1) & 1];
      G.ldv = s.maxh;
      if ((rc = gemm<true>(G, L[l - 1], wk, m, st, who))) return rc;
      in = G.V;
      ldin = G.ldv;
    }
    FitGemm<double> O{};  // output layer: E_i = v_{L-1} . wo + bo
    O.r0 = s.start[t];
    O.n = n;
    O.K = s.w[nlayer - 1];
    O.N = 1;
    O.src[0] = in;
    O.lds[0] = ldin;
    O.nsrc = 1;
    O.wo = pt + s.woff[nlayer];
    fit_out_kernel<double><<<(unsigned)((n + 3) / 4), 128, 0, st>>>(O, O.wo + O.K, E);
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
  layout(s, false, L);
  const WorkMap m = work_map(s, nloc);
  double *buf = reinterpret_cast<double *>(wk + m.buffers);
  const size_t bs = (size_t)nloc * s.maxh;
  double *Z[2] = {buf, buf + bs}, *Sb[2] = {buf + 2 * bs, buf + 3 * bs};
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const double *pt = params + (size_t)t * s.P;
    for (int q = 0; q + 1 < nlayer; ++q)
      if ((rc = split_b(pt + s.woff[nlayer - 1 - q], L[q], false, wk, st, who))) return rc;
    const double *wo = pt + s.woff[nlayer];
    {  // dz of the last hidden layer
      const int K = s.w[nlayer - 1];
      last_dz_kernel<<<(unsigned)std::min<int64_t>(n, 152 * 32), 256, 0, st>>>(s.start[t], n, K, g, wo,
                                                                             act + s.aoff[nlayer - 1], s.H, Z[0],
                                                                             s.maxh);
      if ((rc = launch_status(who))) return rc;
    }
    const double *S = nullptr;  // dE/dv of the layer being walked; NULL: g wo (the last hidden layer)
    int cur = 0;
    for (int l = nlayer - 1; l >= 1; --l) {
      TcGemm G{};
      G.r0 = s.start[t];
      G.n = n;
      G.K = s.w[l];
      G.N = s.w[l - 1];
      G.A = Z[cur];
      G.lda = s.maxh;
      G.skip = s.w[l] == s.w[l - 1];
      G.S = S;
      G.ldS = s.maxh;
      G.g = g;
      G.wo = wo;
      if (l > 1) {
        G.T = act + s.aoff[l - 1];
        G.ldT = s.H;
        G.Snext = Sb[cur];
        G.Z = Z[cur ^ 1];
        G.ldz = s.maxh;
      } else {
        G.out = dD;
        G.ldo = s.w[0];
      }
      if ((rc = gemm<false>(G, L[nlayer - 1 - l], wk, m, st, who))) return rc;
      S = G.Snext;
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
