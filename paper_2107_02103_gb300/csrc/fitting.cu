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
#include "tc_gemm.cuh"

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
  const io_t<real> *W;     // forward: W [K][N] (wt: W [N][K] read as its transpose); backward: W [N][K] transposed
  const io_t<real> *bias;  // forward: [N], NULL (lin only) for none
  bool lin;                // forward: out = acc + bias, no tanh (an output layer of several outputs, or g W^T)
  bool wt;                 // forward: read W as [N][K]
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
    return from_io<real>(P.wt ? P.W[(size_t)nn * P.K + k] : P.W[(size_t)k * P.N + nn]);
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
        if (P.lin)
          v = P.bias ? v + from_io<real>(P.bias[nn]) : v;
        else
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
  int nlayer, ntypes, nout;  // nout = widths[nlayer], the outputs per atom
  int w[DP_MAX_LAYERS + 1];
  int64_t P;       // parameters per type
  int64_t H;       // sum of hidden widths (row length of act)
  int maxh;        // largest hidden width
  int64_t woff[DP_MAX_LAYERS + 1];  // offset of W_l in a type's parameters (l >= 1)
  int64_t aoff[DP_MAX_LAYERS + 1];  // column offset of hidden layer l in act
  int64_t start[DP_MAX_TYPES + 1];
};

// multi: whether the output layer may have several outputs (the FMA-pipe kernels); the tensor-core
// net has one (the energy).
int fit_shape(const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start, FitShape *s,
              bool multi = false) {
  if (!widths || !type_start) return set_error(DP_ERR_NULL, "widths or type_start is NULL");
  if (nlayer < 1 || nlayer > DP_MAX_LAYERS)
    return set_error(DP_ERR_UNSUPPORTED, "nlayer = %d outside [1, %d]", nlayer, DP_MAX_LAYERS);
  if (ntypes < 1 || ntypes > DP_MAX_TYPES)
    return set_error(DP_ERR_UNSUPPORTED, "ntypes = %d outside [1, %d]", ntypes, DP_MAX_TYPES);
  if (!multi && widths[nlayer] != 1)
    return set_error(DP_ERR_SHAPE, "the output layer has width %d, not 1", widths[nlayer]);
  s->nout = widths[nlayer];
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
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s, true);
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
    chain_sources<real>(s, nlayer, D, act, G);
    if (s.nout == 1) {  // E_i = v . wo + bo: a dot product per atom
      G.N = 1;
      G.wo = pt + s.woff[nlayer];
      fit_out_kernel<real><<<(unsigned)((n + 3) / 4), 128, 0, st>>>(G, G.wo + G.K, E);
      rc = launch_status("dp_fitting_fwd");
    } else {  // E_i = v W_out + b_out: a GEMM without tanh
      G.N = s.nout;
      G.W = pt + s.woff[nlayer];
      G.bias = G.W + (size_t)G.K * G.N;
      G.lin = true;
      G.out = E;
      G.ldo = s.nout;
      rc = launch_gemm<real, true>(G, st, "dp_fitting_fwd");
    }
    if (rc) return rc;
  }
  return DP_OK;
}

template <typename real>
int fitting_grad(const io_t<real> *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                 const io_t<real> *act, const io_t<real> *g, io_t<real> *dD, io_t<real> *work, void *stream) {
  clear_error();
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s, true);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (!params || !dD || (s.H > 0 && !act) || ((nlayer > 2 || s.nout > 1) && !work))
    return set_error(DP_ERR_NULL, "dp_fitting_grad: NULL array");
  if (s.nout > 1 && !g) return set_error(DP_ERR_NULL, "dp_fitting_grad: g is NULL for a net of %d outputs", s.nout);
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
    if (s.nout > 1) {  // dE/dv_{nlayer-1} = g W_out^T, [n][nout] x [nout][widths[nlayer-1]], first
      FitGemm<real> Z{};
      Z.r0 = G.r0;
      Z.n = n;
      Z.K = s.nout;
      Z.N = s.w[nlayer - 1];
      Z.src[0] = g;
      Z.lds[0] = s.nout;
      Z.nsrc = 1;
      Z.W = pt + s.woff[nlayer];  // W_out [widths[nlayer-1]][nout], read transposed
      Z.wt = true;
      Z.lin = true;
      Z.out = buf[0];
      Z.ldo = s.maxh;
      if ((rc = launch_gemm<real, true>(Z, st, "dp_fitting_grad"))) return rc;
      S = buf[0];
      ldS = s.maxh;
      cur = 1;
    }
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
// (tc_gemm.cuh: the digit splitting, the split kernels and gemm_kernel)
namespace tc {

// The layer's epilogue over the chunk's n x N outputs, from the shares' partial results summed in
// a fixed order (so a call's results do not depend on timing):
//   forward:  t = tanh(acc + bias); act[row][col] = t; V[row][col] = t (+ A[row][col] when the layer
//             keeps its width: the identity skip, v_l = t_l + v_{l-1})
//   backward: s = acc (+ S[row][col] or g_row wo_col when the layer kept its width); then either
//             out[row][col] = s (dE/dD, the last GEMM) or S_next[row][col] = s and
//             Z[row][col] = s (1 - t_prev^2) with t_prev = T[row][col] (the next GEMM's A)

template <bool kFwd>
__global__ void __launch_bounds__(256) epilogue_kernel(const TcGemm P, int ksplit) {
  // rows over the grid, columns over the block (no 64-bit division per element)
  for (int64_t rc = blockIdx.x; rc < P.n; rc += gridDim.x)
  for (int nn = threadIdx.x; nn < P.N; nn += blockDim.x) {
    const int64_t row = P.r0 + rc;
    Sum3 acc;
    for (int z = 0; z < ksplit; ++z) acc.add(P.part[((size_t)z * P.Mp + rc) * P.Np + nn]);
    double v = acc.value(P.Eexp[rc], P.Fexp[nn]);
    if constexpr (kFwd) {
      if (P.lin) {
        P.V[row * P.ldv + nn] = v + P.bias[nn];
      } else {
        const double t = dfl::tanh_d(v + P.bias[nn]);
        P.act[row * P.ldact + nn] = t;
        P.V[row * P.ldv + nn] = P.skip ? t + P.A[row * P.lda + nn] : t;
      }
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

// dz of the last hidden layer: Z[row][k] = s (1 - t_k^2), t its tanh outputs and s = dE/dv of that layer:
// g_row wo_k (one output) or S[row][k] (several: g W_out^T, made first)
__global__ void __launch_bounds__(256) last_dz_kernel(int64_t r0, int64_t n, int K, const double *__restrict__ g,
                                                      const double *__restrict__ wo, const double *__restrict__ S,
                                                      int64_t ldS, const double *__restrict__ T, int64_t ldT,
                                                      double *__restrict__ Z, int64_t ldz) {
  for (int64_t rr = blockIdx.x; rr < n; rr += gridDim.x)
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int64_t row = r0 + rr;
    const double t = T[row * ldT + k];
    const double sv = S ? S[row * ldS + k] : (g ? g[row] : 1.0) * wo[k];
    Z[row * ldz + k] = sv * fma(-t, t, 1.0);
  }
}

// The GEMMs on the tensor cores: the hidden layers, and with several outputs the output layer too
// (forward: v W_out + b_out; backward: g W_out^T, first).  GEMM q of a direction works on layer
// gemm_layer(s, fwd, q): forward 1 .. L-1 (then L), backward (L, then) L-1 .. 1.
int gemm_count(const FitShape &s) { return s.nlayer - 1 + (s.nout > 1 ? 1 : 0); }
int gemm_layer(const FitShape &s, bool fwd, int q) {
  return fwd ? q + 1 : s.nlayer - q - (s.nout > 1 ? 0 : 1);
}

// Where the B planes and column exponents of each GEMM of one type sit in the work buffer.  After
// them come the A planes and row exponents of one chunk of at most kChunkRows atoms, and the
// [nloc][max hidden width] buffers between layers (forward: 2, backward: 4).
constexpr int64_t kChunkRows = 16384;
struct Layer {
  int K, N, Np, Kp;
  size_t planes, fexp;  // byte offsets
};
size_t layout(const FitShape &s, bool fwd, Layer *out) {
  size_t off = 0;
  for (int q = 0; q < gemm_count(s); ++q) {
    const int l = gemm_layer(s, fwd, q);
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
  Layer L[DP_MAX_LAYERS + 1];
  WorkMap m{};
  m.bplanes = std::max(layout(s, true, L), layout(s, false, L));
  int kmax = 1;
  for (int l = 0; l <= s.nlayer; ++l) kmax = std::max(kmax, s.w[l]);  // every GEMM's K is a layer width
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
  for (int l = 0; l <= s.nlayer; ++l) Npmax = std::max(Npmax, (int)round_up(s.w[l], kTN));
  int64_t part = kTargetCtas * kTM * kTN + m.Mp * Npmax;
  for (int q = 0; q < gemm_count(s); ++q)
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
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s, true);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (!params || !D || !E || (s.H > 0 && !act)) return set_error(DP_ERR_NULL, "%s: NULL array", who);
  if ((rc = check_work(s, nloc, work, work_nbytes, who)) || (rc = set_smem(who))) return rc;
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(work);
  Layer L[DP_MAX_LAYERS + 1];
  layout(s, true, L);
  const WorkMap m = work_map(s, nloc);
  double *V[2] = {reinterpret_cast<double *>(wk + m.buffers), nullptr};
  V[1] = V[0] + (size_t)nloc * s.maxh;
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const double *pt = params + (size_t)t * s.P;
    for (int q = 0; q < gemm_count(s); ++q)  // this type's weights as digit planes (the previous type's are done with)
      if ((rc = split_b(pt + s.woff[gemm_layer(s, true, q)], L[q], true, wk, st, who))) return rc;
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
    if (s.nout == 1) {  // output layer: E_i = v_{L-1} . wo + bo, a dot product per atom (FP64 pipe)
      FitGemm<double> O{};
      O.r0 = s.start[t];
      O.n = n;
      O.K = s.w[nlayer - 1];
      O.N = 1;
      O.src[0] = in;
      O.lds[0] = ldin;
      O.nsrc = 1;
      O.wo = pt + s.woff[nlayer];
      fit_out_kernel<double><<<(unsigned)((n + 3) / 4), 128, 0, st>>>(O, O.wo + O.K, E);
      rc = launch_status(who);
    } else {  // several outputs: E_i = v_{L-1} W_out + b_out, a GEMM on the tensor cores without tanh
      TcGemm G{};
      G.r0 = s.start[t];
      G.n = n;
      G.K = s.w[nlayer - 1];
      G.N = s.nout;
      G.A = in;
      G.lda = ldin;
      G.lin = true;
      G.bias = pt + s.woff[nlayer] + (size_t)G.K * G.N;
      G.V = E;
      G.ldv = s.nout;
      rc = gemm<true>(G, L[nlayer - 1], wk, m, st, who);
    }
    if (rc) return rc;
  }
  return DP_OK;
}

int grad(const double *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
         const double *act, const double *g, double *dD, void *work, size_t work_nbytes, void *stream) {
  clear_error();
  static const char *who = "dp_fitting_grad_tc_f64";
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s, true);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  if (nloc == 0) return DP_OK;
  if (nlayer == 1) return set_error(DP_ERR_UNSUPPORTED, "a fitting net without hidden layers has dD = wo");
  if (!params || !dD || (s.H > 0 && !act)) return set_error(DP_ERR_NULL, "%s: NULL array", who);
  if (s.nout > 1 && !g) return set_error(DP_ERR_NULL, "%s: g is NULL for a net of %d outputs", who, s.nout);
  if ((rc = check_work(s, nloc, work, work_nbytes, who)) || (rc = set_smem(who))) return rc;
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(work);
  Layer L[DP_MAX_LAYERS + 1];
  layout(s, false, L);
  const WorkMap m = work_map(s, nloc);
  double *buf = reinterpret_cast<double *>(wk + m.buffers);
  const size_t bs = (size_t)nloc * s.maxh;
  double *Z[2] = {buf, buf + bs}, *Sb[2] = {buf + 2 * bs, buf + 3 * bs};
  for (int t = 0; t < ntypes; ++t) {
    const int64_t n = s.start[t + 1] - s.start[t];
    if (n == 0) continue;
    const double *pt = params + (size_t)t * s.P;
    for (int q = 0; q < gemm_count(s); ++q)
      if ((rc = split_b(pt + s.woff[gemm_layer(s, false, q)], L[q], false, wk, st, who))) return rc;
    const double *wo = pt + s.woff[nlayer];
    const double *S = nullptr;  // dE/dv of the layer being walked; NULL: g wo (the last hidden layer)
    const int q0 = s.nout > 1 ? 1 : 0;  // the hidden layers' GEMMs come after g W_out^T
    if (s.nout > 1) {  // dE/dv_{nlayer-1} = g W_out^T ([n][nout] x [nout][widths[nlayer-1]], tensor cores),
                       // into Sb[1], which the walk below first writes after its first GEMM has read it
      TcGemm G{};
      G.r0 = s.start[t];
      G.n = n;
      G.K = s.nout;
      G.N = s.w[nlayer - 1];
      G.A = g;
      G.lda = s.nout;
      G.out = Sb[1];
      G.ldo = s.maxh;
      if ((rc = gemm<false>(G, L[0], wk, m, st, who))) return rc;
      S = Sb[1];
    }
    {  // dz of the last hidden layer
      const int K = s.w[nlayer - 1];
      last_dz_kernel<<<(unsigned)std::min<int64_t>(n, 152 * 32), 256, 0, st>>>(s.start[t], n, K, g, wo, S, s.maxh,
                                                                             act + s.aoff[nlayer - 1], s.H, Z[0],
                                                                             s.maxh);
      if ((rc = launch_status(who))) return rc;
    }
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
      if ((rc = gemm<false>(G, L[q0 + nlayer - 1 - l], wk, m, st, who))) return rc;
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
  if (fit_shape(widths, nlayer, 1, ts, &s, true)) return 0;
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

// Device address of the array in the current context.  In host code the array's
// name only stands in for it; the runtime gives the address.  It is looked up
// on every call (the lookup allocates nothing), so that a context made anew --
// after cudaDeviceReset, or on another device -- is served at its own address.
int static_scratch(double **out) {
  void *q = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&q, g_fit_scratch);
  if (e != cudaSuccess)
    return set_error(DP_ERR_CUDA, "dp_fitting_grad_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
  *out = static_cast<double *>(q);
  return DP_OK;
}

int fitting_grad_noalloc(const double *params, const int32_t *widths, int nlayer, int ntypes,
                         const int64_t *type_start, const double *act, const double *g, double *dD, void *stream) {
  clear_error();
  FitShape s{};
  int rc = fit_shape(widths, nlayer, ntypes, type_start, &s, true);
  if (rc) return rc;
  const int64_t nloc = s.start[ntypes];
  const size_t need = (nlayer > 2 || s.nout > 1) ? (size_t)2 * (size_t)nloc * (size_t)s.maxh : 0;
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

// This unit's GEMM wait timeouts (see tc_gemm.cuh), for dp_tc_wait_timeouts.
int take_wait_timeouts_fitting(unsigned int *count) { return tc::take_wait_timeouts(count); }

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
