// Exact f64 GEMMs on the tcgen05 tensor cores, shared by the fitting net and the
// tensor-core form of the tabulated embedding.
#pragma once

#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>

#include "dp_common.cuh"

namespace dpc {
namespace {

// ------------------------------------------------- f64 GEMMs on the tensor cores
// GB300 retires FP64 at 2 lanes per clock per SM but fp16 products on its
// tcgen05 tensor cores at ~1000 times that rate.  An f64 GEMM C = A B is
// recovered from fp16 products by splitting every operand element into base-64
// digits (the error-free splitting of Ozaki et al., here with balanced digits):
//   a_ik = 2^(E_i + 1) sum_{s=1..9} A_s[i][k] 64^-s + r_ik,  A_s integers in [-32, 32],  |r_ik| < 2^(E_i - 53),
// with max_k |a_ik| < 2^E_i: the row's 53-bit fixed point a 2^(53 - E) is truncated toward zero and
// biased by 32 (64^7 + ... + 1); its eight low 6-bit fields less 32 are digits 2 .. 9, and what lies
// above them (an arithmetic shift) is digit 1.  Likewise b_kj with a column exponent F_j, so that
//   C_ij = 2^(E_i + F_j + 2) sum_{d=2..10} 64^-d sum_{s+t=d} (A_s B_t)_ij + (terms with s + t > 10 and the r).
// Every (A_s B_t)_ij is a sum of integer products |A_s B_t| <= 1024; a diagonal
// d has at most 9 of them, so its fp32 sum on the tensor cores is exact while
// a block's share of K is at most kMaxShareK = 1792 (9 x 1792 x 1024 < 2^24).
// The 9 diagonal sums of an output are combined on the FP32 pipe into four
// floats (the two largest by an exact two-sum, the rest in float-float, whose
// rounding lies ~2^-60 below the result); the caller's epilogue (Sum3 below)
// adds the shares' floats into a three-float sum by exact two-sums and
// converts it to f64 once -- or, in the tabulation's GEMMs, recombines the
// diagonals exactly as one 128-bit integer and rounds that once (diag_s128,
// s128_to_f64).  The tabulation's backward, whose K is M1 <= 144, splits into
// seven 8-bit digits instead (Digits7x8; 28 products, diag7_to_f64).
// What rounds is that conversion, the 53-bit truncation of the operands and
// the dropped terms: |error| <~ K 2^-49 max_k|a_ik| max_k|b_kj|, against
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
// digit products as 13 MMAs (M 128, K 16, fp16 in, fp32 accumulators in TMEM,
// one 48-column block per diagonal; digit s of A against all of B's digits
// t <= 8 - s at once, N up to 240) and commits them to the stage's "empty" mbarrier, which
// the producer waits on before refilling the stage.  A last commit on a
// barrier used once releases the four warps, which read their TMEM lane
// quadrant (rows), combine the diagonals and write the share's result as four
// floats; the caller's epilogue kernel sums the shares in a fixed order,
// scales by 2^(E+F) and finishes the outputs.  Two optional modes serve sparse
// operands (the tabulated embedding's interval moments): a per-tile list of the
// K slices in use (the others are zero and are skipped; the shares then cut the
// used slices, and a tile whose used slices fit one share can write its f64
// outputs itself), and per-tile slice flags that skip unwanted output tiles,
// whose wanted outputs are scattered to per-run slots instead of a dense array.
// Every wait on an mbarrier is bounded; a wait that gives up makes the tile's
// outputs NaN (the accumulators are not read) and counts one timeout in
// g_wait_timeouts, which the host reads through dp_tc_wait_timeouts.
namespace tc {
constexpr int kS = 9;      // digits per operand element
constexpr int kBits = 6;   // bits per digit
constexpr int kFrac = kS * kBits - 1;  // 53 fractional bits; the ninth digit's spare bit keeps the balanced top digit in range
constexpr int kPad = kS * kBits - kFrac;  // a digit vector stands for 2^(E + kPad) sum_s d_s 64^-s
// 32 (64^7 + ... + 1): added to a fixed point f in (-2^53, 2^53), it makes each of the eight low 6-bit
// fields a digit plus 32 and leaves floor((f + bias) / 64^8) in [-32, 32] as the top digit
constexpr int64_t kDigitBias = 32ll * ((1ll << 48) - 1ll) / 63ll;
constexpr int kTM = 128, kTN = 48, kTK = 16;  // CTA tile; K per stage (one MMA)
constexpr int kStages = 4;
constexpr int kThreads = 128;  // one warp per TMEM lane quadrant; lane 0 of warps 0 and 1: producer and MMA issuer
constexpr int kMaxShareK = 1792;
constexpr int kNonFinite = 1 << 20;  // exponent of a row or column holding inf or NaN
constexpr uint32_t kLBO = 128, kSBO = 256;  // core matrices: next along K at +128 B, next 8 rows at +256 B
constexpr int kPlaneA = kTM * kTK * 2, kPlaneB = kTN * kTK * 2;  // bytes of one digit plane in a stage
constexpr int kStageBytes = kS * (kPlaneA + kPlaneB);
constexpr uint32_t kTmemCols = 512;  // allocation (a power of two); kS * kTN = 432 used
constexpr int kMaxShareSlices = kMaxShareK / kTK;
constexpr size_t kSmemTail = (size_t)kStages * kStageBytes + (2 * kStages + 1) * 8 + 16;  // used-slice list
constexpr int kScatKeys = kTM / 4 + 1, kScatAtoms = kTN / 4;  // scatter: keys (kq >= 4) and atoms of a tile
constexpr size_t kSmemTotal = kSmemTail + (kMaxShareSlices + 2) * 4 + kScatKeys * kScatAtoms * 4;
static_assert((size_t)kS * kMaxShareK * 32 * 32 < (1u << 24), "fp32 diagonal sums must stay exact");
static_assert(kDigitBias < (1ll << 48) && kFrac == 53 && kS == 9, "top digit floor((f + bias) / 2^48) within [-32, 32]");
static_assert(kMaxShareK % kTK == 0 && kS * kTN <= (int)kTmemCols, "shares and TMEM");
static_assert(kSmemTotal <= 227 * 1024, "shared memory per block");

__host__ __device__ constexpr int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

__device__ __forceinline__ int exp_bits(double x) { return (int)(((uint64_t)__double_as_longlong(x) >> 52) & 0x7ff); }
// E with max |x| < 2^E from the largest biased exponent (normal x: |x| < 2^(eb - 1022))
__device__ __forceinline__ int exp_of_max(int ebmax) { return ebmax == 0x7ff ? kNonFinite : max(ebmax, 1) - 1022; }

// A digit scheme: NS balanced digits of NB bits (digit 1 in [-2^(NB-1), 2^(NB-1)], the others in
// [-2^(NB-1), 2^(NB-1) - 1]) for an element's NS NB - 1 fractional bits.  The tensor-core GEMMs use 9 x 6
// bits (kS, kBits: a share of K up to kMaxShareK = 1792) or, where K <= 144, 7 x 8 bits (products up to
// 2^14, seven of them on a diagonal: 7 x 2^14 x 144 < 2^24), which needs 28 digit products instead of 45.
template <int NS, int NB>
struct Digits {
  static constexpr int kNS = NS, kNB = NB;
  static constexpr int kFrac = NS * NB - 1;
  static constexpr int kPad = NS * NB - kFrac;  // a digit vector stands for 2^(E + kPad) sum_s d_s 2^(-NB s)
  static constexpr int64_t kBias = (1ll << (NB - 1)) * ((1ll << (NB * (NS - 1))) - 1ll) / ((1ll << NB) - 1ll);
  static constexpr uint32_t kHalf = 1u << (NB - 1);
  // the fp16 pair 1024 + kHalf: field u in [0, 2^NB] is encoded as 0x6400 | u (1024 + u) and this comes off
  static constexpr uint32_t kOffPair = (0x6400u + kHalf) * 0x10001u;
  static_assert(kBias < (1ll << (NB * (NS - 1))) && NB * (NS - 1) <= 56 && NB <= 9, "balanced top digit in range");
};
using Digits9x6 = Digits<9, 6>;
using Digits7x8 = Digits<7, 8>;
static_assert(Digits9x6::kBias == kDigitBias && Digits9x6::kFrac == kFrac && Digits9x6::kPad == kPad, "the 9 x 6 scheme");
static_assert(Digits7x8::kFrac == 55 && Digits7x8::kPad == 1 && Digits7x8::kBias < (1ll << 48), "the 7 x 8 scheme");

// x 2^(kFrac - E) truncated toward zero (|x| < 2^E, so |.| < 2^kFrac), plus the scheme's bias (see digit_pairs)
template <class D = Digits9x6>
__device__ __forceinline__ int64_t biased_fixed(double x, int E) {
  const uint64_t b = (uint64_t)__double_as_longlong(x);
  const int eb = (int)((b >> 52) & 0x7ff);
  const uint64_t mant = b & 0xfffffffffffffull;
  const uint64_t m = eb ? (mant | (1ull << 52)) : mant;
  const int sh = (eb ? eb - 1075 : -1074) - E + D::kFrac;  // |x| 2^(kFrac - E) = m 2^sh, sh <= kFrac - 53 for finite x
  const int64_t mag = (int64_t)(sh >= 0 ? m << min(sh, 10) : (sh > -64 ? m >> -sh : 0ull));
  return (b >> 63 ? -mag : mag) + D::kBias;
}

// The NS balanced digits of two elements from their biased fixed points g, digit s of both packed as an
// fp16 pair (element 0 in the low half): field u in [0, 2^NB] (digit + 2^(NB-1)) is encoded as 0x6400 | u,
// the fp16 1024 + u, and 1024 + 2^(NB-1) comes off exactly.  Digits 2 .. NS are the low NB-bit fields;
// digit 1 is g shifted right by NB (NS - 1).
template <class D = Digits9x6>
__device__ __forceinline__ void digit_pairs(int64_t g0, int64_t g1, uint32_t (&h)[D::kNS]) {
  constexpr int NS = D::kNS, NB = D::kNB;
  constexpr uint32_t kMask = (1u << NB) - 1;
#pragma unroll
  for (int s = 1; s <= NS; ++s) {
    const int sh = NB * (NS - s);
    const uint32_t d0 = s == 1 ? (uint32_t)((g0 >> sh) + D::kHalf) : (uint32_t)(g0 >> sh) & kMask;
    const uint32_t d1 = s == 1 ? (uint32_t)((g1 >> sh) + D::kHalf) : (uint32_t)(g1 >> sh) & kMask;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(h[s - 1]) : "r"(0x64006400u | d0 | (d1 << 16)), "r"(D::kOffPair));
  }
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
template <class D>
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
  constexpr int NS = D::kNS;
  const size_t plane = (size_t)RT * kTK * 2, block = NS * plane;
  const int ri = (int)(r % RT);
  unsigned char *rowbase = planes + (size_t)(r / RT) * (Kp / kTK) * block + (ri >> 3) * kSBO + (ri & 7) * 16 + kp * 4;
  for (int k0 = kc * kSplitK; k0 < min(Kp, kc * kSplitK + kSplitK); k0 += 8) {
    const int k = k0 + 2 * kp;
    const double x0 = x(k), x1 = x(k + 1);
    uint32_t h[NS];
    digit_pairs<D>(biased_fixed<D>(x0, E), biased_fixed<D>(x1, E), h);
    unsigned char *dst = rowbase + (size_t)(k0 / kTK) * block + ((k0 % kTK) >> 3) * kLBO;
#pragma unroll
    for (int s = 0; s < NS; ++s) *reinterpret_cast<uint32_t *>(dst + s * plane) = h[s];
  }
}

// f 2^e as a double, exactly, by moving fields (f finite; |e| < 900, so a normal result stays normal
// and a float that is zero stays zero; float subnormals, which the sums do not produce, widen to 0)
__device__ __forceinline__ double widen_pow2(float f, int e) {
  const double d = dfl::widen(f);
  const long long b = __double_as_longlong(d);
  return (b & 0x7fffffffffffffffll) ? __longlong_as_double(b + ((long long)e << 52)) : d;
}

// The shares' results of one output summed in a fixed order: each share's four floats are added
// into a three-float sum by exact two-sums on the FP32 pipe (only the last component rounds, ~2^-72
// below the sum), which is converted to f64 once and scaled by the row and column powers of two.
struct Sum3 {
  float s0 = 0.f, s1 = 0.f, s2 = 0.f;
  __device__ __forceinline__ void add(float x) {
    float t = __fadd_rn(s0, x), z = __fsub_rn(t, s0);
    const float e0 = __fadd_rn(__fsub_rn(s0, __fsub_rn(t, z)), __fsub_rn(x, z));
    s0 = t;
    t = __fadd_rn(s1, e0);
    z = __fsub_rn(t, s1);
    const float e1 = __fadd_rn(__fsub_rn(s1, __fsub_rn(t, z)), __fsub_rn(e0, z));
    s1 = t;
    s2 = __fadd_rn(s2, e1);
  }
  __device__ __forceinline__ void add(const float4 q) {
    add(q.x);
    add(q.y);
    add(q.z);
    add(q.w);
  }
  // the sum times 2^(E + F); NaN for a row or column with an inf or NaN, or a NaN share
  __device__ __forceinline__ double value(int E, int F) const {
    if (E >= kNonFinite || F >= kNonFinite || s0 != s0) return __longlong_as_double(0x7ff8000000000000ll);
    const int e = E + F + 2 * kPad;
    if (e > -900 && e < 900)  // the scaling moves exponent fields only (sums stay normal)
      return __dadd_rn(__dadd_rn(widen_pow2(s0, e), widen_pow2(s1, e)), widen_pow2(s2, e));
    return scalbn(__dadd_rn(__dadd_rn(dfl::widen(s0), dfl::widen(s1)), dfl::widen(s2)), e);
  }
};

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
  // sparse operands (NULL for dense ones)
  const unsigned char *kocc;  // [Np / kTN][Kp / kTK]: nonzero where the B tile has a nonzero entry in the
                              // slice; share z of a tile then takes its used slices z S .. z S + S - 1
                              // (S = slices_per_split), and a share past its last used slice writes nothing
  const unsigned char *sflags;  // [Np / kTN][nsf]: flags of the K slices the atoms of a B tile use; output
                                // tile (x, y) is wanted when one of slices 8 y .. 8 y + 7 is flagged
  int nsf;
  // scatter (with sflags): output (row kq key + q, column 4 a + k), q < 6 <= kq, key < nkeys, a < natoms,
  // goes to scat[(a cap + slot) 24 + 6 k + q] when atom atom0 + a has type alpha (atype clamped into
  // [0, ntypes)) and key is keys[(atom0 + a) cap + slot] for a slot < nslots[atom0 + a]; nothing is
  // written to part
  float4 *scat;
  const short *keys;
  const int *nslots;
  const int32_t *atype;
  int64_t natoms, atom0;
  int nkeys, cap, alpha, ntypes, kq;
  // direct output (with kocc): a tile whose used slices fit one share writes its outputs as f64,
  // scaled by 2^(E_row + F_col), to tout[((atom0 + a) 4 + k) ldt + row] for row < ldt and the atoms
  // a < natoms of type alpha, and nothing to part (the forward tabulation's T)
  double *tout;
  int ldt;
  bool skip;
  // forward
  bool lin;  // an output layer of several outputs: V[row][col] = acc + bias, no tanh, act unused
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

// Bounded mbarrier waits that gave up, one count per CTA (this translation unit's kernels).
__device__ unsigned int g_wait_timeouts;

// The count, read after a device synchronisation, then cleared.
int take_wait_timeouts(unsigned int *count) {
  unsigned int v = 0, zero = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpyFromSymbol(&v, g_wait_timeouts, sizeof v);
  if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_wait_timeouts, &zero, sizeof zero);
  if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_tc_wait_timeouts: %s", cudaGetErrorString(e));
  *count += v;
  return DP_OK;
}

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  uint32_t done = 0;
  for (int it = 0; it < (1 << 24) && !done; ++it)
    asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
                 : "=r"(done)
                 : "r"(bar), "r"(parity)
                 : "memory");
  return done != 0;
}

// sum_d v[d][c] 64^-(d+2) (the diagonal sums of one output, read from TMEM) as four floats on the FP32
// pipe: diagonals 2 and 3 (d = 0, 1) as an exact two-sum, 4 .. 10 in float-float, smallest first (its
// rounding lies ~2^-60 below the sum).
template <int W>
__device__ __forceinline__ float4 diag_combine_w(const float (&v)[kS][W], int c) {
  dfl::df64 lo(0.0f);
#pragma unroll
  for (int d = kS - 1; d >= 2; --d) {
    const float x = v[d][c] * __uint_as_float((uint32_t)(127 - kBits * (d + 2)) << 23);  // exact: 64^-(d+2)
    lo = lo + dfl::df64(x);
  }
  const float a = v[0][c] * 0x1p-12f, b = v[1][c] * 0x1p-18f;  // exact
  const float s = __fadd_rn(a, b), bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return make_float4(s, e, lo.hi, lo.lo);
}
__device__ __forceinline__ float4 diag_combine(const float (&v)[kS][8], int c) { return diag_combine_w<8>(v, c); }
__device__ __forceinline__ float4 diag_combine4(const float (&v)[kS][4], int c) { return diag_combine_w<4>(v, c); }

// A float that holds an integer below 2^24 in magnitude (a diagonal sum) as an int: exact.
__device__ __forceinline__ int exact_int(float f) { return __float2int_rz(f); }

// The nine diagonal sums of one output (exact integers below 2^24; diagonal d weighs 64^-(d+2)) as one
// exact integer in units of 2^-60, S = sum_d v[d][c] 2^(6 (8 - d)), |S| < 2^74: integer adds, no rounding.
template <int W>
__device__ __forceinline__ __int128 diag_int(const float (&v)[kS][W], int c) {
  static_assert(kS == 9 && kBits == 6, "the integer recombination assumes nine 6-bit digits");
  long long lo = 0;  // diagonals 4 .. 10: below 2^24 2^36 64/63 < 2^61
#pragma unroll
  for (int d = 2; d < kS; ++d) lo += (long long)exact_int(v[d][c]) << (kBits * (kS - 1 - d));
  const long long hi = (long long)exact_int(v[0][c]) * 64 + exact_int(v[1][c]);  // diagonals 2, 3 over 2^42
  return ((__int128)hi << 42) + lo;
}

// diag_int for diagonal sums below 2^22 in magnitude: each converts to int by one FP32 add of
// 1.5 2^23 (the sum's integer lands in the low significand bits exactly) and one integer subtract.
template <int W>
__device__ __forceinline__ __int128 diag_int_small(const float (&v)[kS][W], int c) {
  auto to_int = [](float f) { return __float_as_int(__fadd_rn(f, 12582912.0f)) - 0x4B400000; };
  long long lo = 0;
#pragma unroll
  for (int d = 2; d < kS; ++d) lo += (long long)to_int(v[d][c]) << (kBits * (kS - 1 - d));
  const long long hi = (long long)to_int(v[0][c]) * 64 + to_int(v[1][c]);
  return ((__int128)hi << 42) + lo;
}

// S 2^e2 rounded once to the nearest f64 (ties to even), from its bits: integer operations only, except
// where the result falls outside the normal range (never for these sums in practice).
__device__ __forceinline__ double i128_to_double(__int128 S, int e2) {
  if (S == 0) return 0.0;
  const bool neg = S < 0;
  const unsigned __int128 U = neg ? (unsigned __int128)(-S) : (unsigned __int128)S;
  const unsigned long long uh = (unsigned long long)(U >> 64), ul = (unsigned long long)U;
  const int n = uh ? 128 - __clzll((long long)uh) : 64 - __clzll((long long)ul);  // bit length of |S|
  int ex = n - 1 + e2;  // exponent of the leading bit
  unsigned long long m;
  if (n <= 53) {
    m = ul << (53 - n);
  } else {
    const int sh = n - 53;
    m = (unsigned long long)(U >> sh);
    const unsigned long long rem = ul & ((1ull << sh) - 1ull), half = 1ull << (sh - 1);
    if (rem > half || (rem == half && (m & 1ull))) {
      ++m;
      if (m == (1ull << 53)) {
        m >>= 1;
        ++ex;
      }
    }
  }
  if (ex < -1022 || ex > 1023) return (neg ? -1.0 : 1.0) * scalbn((double)m, ex - 52);
  return __longlong_as_double((long long)(((unsigned long long)neg << 63) | ((unsigned long long)(ex + 1023) << 52) |
                                          (m & ((1ull << 52) - 1ull))));
}

// An output from its exact integer: NaN for a row or column with an inf or NaN.
__device__ __forceinline__ double output_value(__int128 S, int E, int F) {
  if (E >= kNonFinite || F >= kNonFinite) return __longlong_as_double(0x7ff8000000000000ll);
  return i128_to_double(S, E + F + 2 * kPad - 2 * kBits - kBits * (kS - 1));
}

// The exponent offset of output_value: an output is S 2^(E + F + kOutExp).
constexpr int kOutExp = 2 * kPad - 2 * kBits - kBits * (kS - 1);

// S 2^(E + F + X) rounded once to the nearest double (ties to even), S the two's complement pair (hi, lo)
// with |S| < 2^126, without branches: |S| is normalised by its leading-zero count, the top 53 bits are
// rounded from the round bit and the sticky bits, and the exponent is added into the bit pattern, so a
// rounding carry moves into it.  Sets `rare` where the result falls outside the normal range (never with
// these operands; the caller then takes output_value), NaN for a row or column with an inf or NaN.
template <int X>
__device__ __forceinline__ double s128_to_f64(long long hi, unsigned long long lo, int E, int F, bool &rare) {
  const unsigned long long sg = (unsigned long long)(hi >> 63);  // all ones when S < 0
  const unsigned long long ml = (lo ^ sg) - sg;                   // |S|, low word
  const unsigned long long mh = ((unsigned long long)hi ^ sg) + (sg & (ml == 0 ? 1ull : 0ull));
  const bool top = mh != 0;
  const int lz = top ? __clzll((long long)mh) : 64 + __clzll((long long)ml);
  const unsigned long long hN = top ? mh : ml, lN = top ? ml : 0ull;
  const int s1 = lz & 63;
  const unsigned long long N = (hN << s1) | ((lN >> 1) >> (63 - s1));  // the leading 64 bits
  const unsigned long long rest = lN << s1;
  const unsigned long long mant = N >> 11;
  const unsigned long long inc = ((N >> 10) & 1ull) & ((((N & 0x3ffull) | rest) != 0 ? 1ull : 0ull) | (mant & 1ull));
  const int ex = 127 - lz + E + F + X;  // exponent of the leading bit
  unsigned long long bits = (((unsigned long long)(ex + 1022) << 52) + mant + inc) | (sg << 63);
  const bool nonfinite = E >= kNonFinite || F >= kNonFinite, zero = lz == 128;
  rare |= !nonfinite && !zero && (unsigned)(ex + 1022) > 2045u;
  bits = zero ? 0ull : bits;
  bits = nonfinite ? 0x7ff8000000000000ull : bits;
  return __longlong_as_double((long long)bits);
}

// output_value without branches, for the wide epilogues: the nine diagonal sums become
// S = T 2^36 + M 2^18 + L (T, M, L each three diagonals, |.| < 2^36.03) as a 128-bit two's complement
// pair, rounded by s128_to_f64.  Equal to output_value(diag_int(v, c), E, F) except where `rare` is set:
// the caller then takes output_value for the group, after all of its outputs, so that no call or branch
// sits between their independent instruction chains (measured: a call site inside each conversion made
// it 3.5 times slower).
template <int W>
__device__ __forceinline__ void diag_s128(const float (&v)[kS][W], int c, long long &hi, unsigned long long &lo) {
  static_assert(kS == 9 && kBits == 6, "three groups of three 6-bit diagonals");
  int x[kS];
#pragma unroll
  for (int d = 0; d < kS; ++d) x[d] = exact_int(v[d][c]);
  const long long T = (long long)x[0] * 4096 + (long long)x[1] * 64 + x[2];
  const long long M = (long long)x[3] * 4096 + (long long)x[4] * 64 + x[5];
  const long long L = (long long)x[6] * 4096 + (long long)x[7] * 64 + x[8];
  const long long A = M * 262144 + L;  // |A| < 2^55
  const unsigned long long tl = (unsigned long long)T << 36;
  lo = tl + (unsigned long long)A;
  hi = (T >> 28) + (A >> 63) + (lo < tl ? 1 : 0);
}
template <int W>
__device__ __forceinline__ double diag_to_f64(const float (&v)[kS][W], int c, int E, int F, bool &rare) {
  long long hi;
  unsigned long long lo;
  diag_s128(v, c, hi, lo);
  return s128_to_f64<kOutExp>(hi, lo, E, F, rare);
}

// The 7 x 8-bit scheme (Digits7x8): seven diagonal sums, diagonal d weighing 256^-(d+2), as one exact
// integer S = sum_d v[d][c] 2^(8 (6 - d)), |S| < 2^72.01; an output is S 2^(E + F + kOutExp7x8).
constexpr int kOutExp7x8 = 2 * Digits7x8::kPad - 2 * 8 - 8 * 6;
template <int W>
__device__ __forceinline__ __int128 diag7_int(const float (&v)[7][W], int c) {
  long long A = 0;  // diagonals 3 .. 6: below 2^24 2^24 256/255 < 2^49
#pragma unroll
  for (int d = 3; d < 7; ++d) A += (long long)exact_int(v[d][c]) << (8 * (6 - d));
  const long long T = (long long)exact_int(v[0][c]) * 65536 + (long long)exact_int(v[1][c]) * 256 + exact_int(v[2][c]);
  return ((__int128)T << 32) + A;
}
template <int W>
__device__ __forceinline__ double diag7_to_f64(const float (&v)[7][W], int c, int E, int F, bool &rare) {
  int x[7];
#pragma unroll
  for (int d = 0; d < 7; ++d) x[d] = exact_int(v[d][c]);
  const long long T = (long long)x[0] * 65536 + (long long)x[1] * 256 + x[2];  // |T| < 2^40.01
  const long long A = (long long)x[3] * 16777216 + (long long)x[4] * 65536 + (long long)x[5] * 256 + x[6];  // < 2^48.01
  const unsigned long long tl = (unsigned long long)T << 32;
  const unsigned long long lo = tl + (unsigned long long)A;
  const long long hi = (T >> 32) + (A >> 63) + (lo < tl ? 1 : 0);
  return s128_to_f64<kOutExp7x8>(hi, lo, E, F, rare);
}
__device__ __forceinline__ double output_value7(__int128 S, int E, int F) {
  if (E >= kNonFinite || F >= kNonFinite) return __longlong_as_double(0x7ff8000000000000ll);
  return i128_to_double(S, E + F + kOutExp7x8);
}

// The rare case of diag_to_f64 / diag7_to_f64 (a result outside the normal range), out of line so that
// the epilogue loops stay small: one output from its diagonal sums (the seventh to ninth unused by the
// 7 x 8 scheme).
__device__ __noinline__ double output_value_rare(float v0, float v1, float v2, float v3, float v4, float v5, float v6,
                                                 float v7, float v8, int E, int F, bool seven) {
  if (seven) {
    const float v[7][1] = {{v0}, {v1}, {v2}, {v3}, {v4}, {v5}, {v6}};
    return output_value7(diag7_int(v, 0), E, F);
  }
  const float v[kS][1] = {{v0}, {v1}, {v2}, {v3}, {v4}, {v5}, {v6}, {v7}, {v8}};
  return output_value(diag_int(v, 0), E, F);
}

__global__ void __launch_bounds__(kThreads, 1) gemm_kernel(const TcGemm P) {
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + kStages * kStageBytes);  // stage loaded
  uint64_t *empty = full + kStages;                                               // stage's MMAs done
  uint64_t *done = empty + kStages;                                               // every MMA done (one use)
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(done + 1);
  int *flags = reinterpret_cast<int *>(tmem_holder + 1);                          // producer / issuer ok
  int *slist = reinterpret_cast<int *>(smem + kSmemTail);  // used slices, their count, the tile's total
  int *stab = slist + kMaxShareSlices + 2;  // scatter: slot of (key, atom) of the tile, or -1; direct: atom wanted
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t m0 = (int64_t)blockIdx.y * kTM;
  const int n0 = blockIdx.x * kTN;
  const int nslices = P.Kp / kTK;
  const int i0 = blockIdx.z * P.slices_per_split;
  if (P.sflags) {  // an output tile no atom of the B tile uses is skipped (uniform)
    const unsigned char *f = P.sflags + (size_t)blockIdx.x * P.nsf;
    const int lo = (int)(m0 / kTK), hi = min(P.nsf, (int)((m0 + kTM) / kTK));
    bool any = false;
    for (int x = lo; x < hi; ++x) any |= f[x] != 0;
    if (!any) return;
  }
  if (P.scat) {  // the tile's slots: (key of the tile, atom) -> slot, or -1
    int *nsa = slist;  // the slot count of each atom of the tile (0: not of type alpha); slist is free here
    for (int x = tid; x < kScatKeys * kScatAtoms; x += kThreads) stab[x] = -1;
    if (tid < kScatAtoms) {
      const int64_t a = (int64_t)(n0 / 4) + tid, i = P.atom0 + a;
      nsa[tid] = a < P.natoms && (!P.atype || clampi(P.atype[i], 0, P.ntypes - 1) == P.alpha) ? P.nslots[i] : 0;
    }
    __syncthreads();
    const int key0 = (int)(m0 / P.kq);
    for (int al = warp; al < kScatAtoms; al += kThreads / 32) {  // a warp per atom, its lanes over the slots
      const short *keys = P.keys + (P.atom0 + n0 / 4 + al) * P.cap;
      for (int slot = lane; slot < nsa[al]; slot += 32) {
        const int key = keys[slot];
        if (key >= key0 && key < key0 + kScatKeys) stab[(key - key0) * kScatAtoms + al] = slot;
      }
    }
  }
  if (P.tout)
    for (int x = tid; x < kScatAtoms; x += kThreads) {
      const int64_t a = (int64_t)(n0 / 4) + x;
      stab[x] = a < P.natoms && (!P.atype || clampi(P.atype[P.atom0 + a], 0, P.ntypes - 1) == P.alpha);
    }
  int nsl = min(nslices - i0, P.slices_per_split);  // dense: > 0, no empty share
  if (P.kocc) {
    // this share's used slices, in order, by a ballot over the tile's flags
    if (warp == 0) {
      const unsigned char *occ = P.kocc + (size_t)blockIdx.x * nslices;
      const int last = i0 + P.slices_per_split;
      int rank = 0;
      for (int b = 0; b < nslices && (rank < last || P.tout); b += 32) {  // uniform; direct output counts all
        const int i = b + lane;
        const bool used = i < nslices && occ[i] != 0;
        const unsigned m = __ballot_sync(0xffffffffu, used);
        const int r = rank + __popc(m & ((1u << lane) - 1u));
        if (used && r >= i0 && r < last) slist[r - i0] = i;
        rank += __popc(m);
      }
      if (lane == 0) {
        slist[kMaxShareSlices] = min(max(rank - i0, 0), P.slices_per_split);
        slist[kMaxShareSlices + 1] = rank;
      }
    }
    __syncthreads();
    nsl = slist[kMaxShareSlices];
    if (nsl == 0) return;  // uniform: no slice left for this share
  }
  const bool direct = P.tout && P.kocc && slist[kMaxShareSlices + 1] <= P.slices_per_split;

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
    for (int j = 0; j < nsl && ok; ++j) {
      const int sl = P.kocc ? slist[j] : i0 + j;
      const unsigned char *asrc = P.aplanes + ((size_t)blockIdx.y * nslices + sl) * (kS * kPlaneA);
      const unsigned char *bsrc = P.planes + ((size_t)blockIdx.x * nslices + sl) * (kS * kPlaneB);
      const int st = j % kStages;
      if (j >= kStages) ok = mbar_wait(smem_u32(empty + st), (uint32_t)((j / kStages - 1) & 1));
      if (!ok) break;
      const uint32_t bar = smem_u32(full + st), dst = sbase + st * kStageBytes;
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"((uint32_t)kStageBytes)
                   : "memory");
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                   "l"(asrc), "r"((uint32_t)(kS * kPlaneA)), "r"(bar)
                   : "memory");
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                       dst + kS * kPlaneA),
                   "l"(bsrc), "r"((uint32_t)(kS * kPlaneB)), "r"(bar)
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
  ok = __syncthreads_and(ok) != 0;  // one answer for the CTA: its accumulators are read only if every wait ended
  if (!ok && tid == 0) atomicAdd(&g_wait_timeouts, 1u);
  asm volatile("tcgen05.fence::after_thread_sync;");

  // combine the diagonals of row 32 (warp % 4) + lane (the warp's TMEM lane quadrant), the warp's
  // third of the columns, 8 at a time
  const int rl = 32 * (warp & 3) + lane;
  float4 *outp = P.scat ? nullptr : P.part + ((size_t)blockIdx.z * P.Mp + m0 + rl) * P.Np + n0;
  const int key = P.scat ? (int)((m0 + rl) / P.kq) : 0, q = P.scat ? (int)(m0 + rl - (int64_t)key * P.kq) : 0;
  const int key_l = P.scat ? key - (int)(m0 / P.kq) : 0;  // this thread's row's key, in the tile
  const bool row_wanted = P.scat && q < 6 && key < P.nkeys;
  const int Erow = direct && m0 + rl < P.ldt ? P.Eexp[m0 + rl] : 0;
  const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
  constexpr int kColsPerWarp = kTN / (kThreads / 128);
  static_assert(kColsPerWarp % 8 == 0, "column share");
#pragma unroll 1
  for (int c0 = (warp >> 2) * kColsPerWarp; c0 < (warp >> 2) * kColsPerWarp + kColsPerWarp; c0 += 8) {
    float v[kS][8];
    if (ok) {  // uniform over the CTA
#pragma unroll
      for (int d = 0; d < kS; ++d)
        asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                     : "=f"(v[d][0]), "=f"(v[d][1]), "=f"(v[d][2]), "=f"(v[d][3]), "=f"(v[d][4]), "=f"(v[d][5]),
                       "=f"(v[d][6]), "=f"(v[d][7])
                     : "r"(trow + (uint32_t)(d * kTN + c0)));
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
    } else {
#pragma unroll
      for (int d = 0; d < kS; ++d)
#pragma unroll
        for (int c = 0; c < 8; ++c) v[d][c] = 0.0f;
    }
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      // The scaling by 2^(E+F+2 kPad), and all f64 arithmetic, is left to the epilogue (or, for a direct
      // output, to the two f64 adds below).
      const float4 val = ok ? diag_combine(v, c) : make_float4(__int_as_float(0x7fc00000), 0.f, 0.f, 0.f);
      if (direct) {
        if (m0 + rl < P.ldt && stab[(c0 + c) >> 2]) {
          Sum3 acc;
          acc.add(val);
          const int64_t a = (int64_t)(n0 >> 2) + ((c0 + c) >> 2);
          P.tout[((P.atom0 + a) * 4 + ((c0 + c) & 3)) * P.ldt + m0 + rl] = acc.value(Erow, P.Fexp[n0 + c0 + c]);
        }
      } else if (outp) {
        outp[c0 + c] = val;
      } else if (row_wanted) {
        const int al = (c0 + c) >> 2, k = (c0 + c) & 3;  // the tile's atom, its column k
        const int slot = stab[key_l * kScatAtoms + al];
        if (slot >= 0) P.scat[((size_t)((n0 >> 2) + al) * P.cap + slot) * 24 + 6 * k + q] = val;
      }
    }
  }

  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

int set_smem(const char *who) {
  static std::atomic<bool> done{false};
  if (done.load(std::memory_order_acquire)) return DP_OK;
  const cudaError_t e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemTotal);
  if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
  done.store(true, std::memory_order_release);
  return DP_OK;
}

// split_rows_kernel with the row exponents found in the same kernel: one warp per group of 8 rows and
// all of K (lane = (row ri8 = lane / 4, pair of k kp = lane % 4)), a first pass over the rows for their
// largest exponents (reduced over the row's four lanes), a second for the digits.  For short rows
// (the tabulation's dT^T, K = M1), where a launch per pass costs more than the passes.
template <class D>
__global__ void __launch_bounds__(128) split_rows_1k_kernel(const double *__restrict__ X, int64_t ld_r, int64_t ld_k,
                                                            int64_t nrows, int K, int64_t rows_p, int Kp, int RT,
                                                            unsigned char *__restrict__ planes, int *__restrict__ exps) {
  constexpr int NS = D::kNS;
  const int lane = threadIdx.x & 31, ri8 = lane >> 2, kp = lane & 3;
  const int64_t g = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);  // 8-row group
  if (g * 8 >= rows_p) return;                                      // warp-uniform
  const int64_t r = g * 8 + ri8;
  const double *__restrict__ xr = X + (r < nrows ? r : 0) * ld_r;
  auto x = [&](int k) { return (r < nrows && k < K) ? __ldg(xr + k * ld_k) : 0.0; };
  int eb = 0;
  for (int k0 = 0; k0 < Kp; k0 += 8) eb = max(eb, max(exp_bits(x(k0 + 2 * kp)), exp_bits(x(k0 + 2 * kp + 1))));
  eb = max(eb, __shfl_xor_sync(0xffffffffu, eb, 1));
  eb = max(eb, __shfl_xor_sync(0xffffffffu, eb, 2));
  const int E = exp_of_max(eb);
  if (kp == 0) exps[r] = E;
  const size_t plane = (size_t)RT * kTK * 2, block = NS * plane;
  const int ri = (int)(r % RT);
  unsigned char *rowbase = planes + (size_t)(r / RT) * (Kp / kTK) * block + (ri >> 3) * kSBO + (ri & 7) * 16 + kp * 4;
  for (int k0 = 0; k0 < Kp; k0 += 8) {
    const int k = k0 + 2 * kp;
    uint32_t h[NS];
    digit_pairs<D>(biased_fixed<D>(x(k), E), biased_fixed<D>(x(k + 1), E), h);
    unsigned char *dst = rowbase + (size_t)(k0 / kTK) * block + ((k0 % kTK) >> 3) * kLBO;
#pragma unroll
    for (int s = 0; s < NS; ++s) *reinterpret_cast<uint32_t *>(dst + s * plane) = h[s];
  }
}

template <class D>
int split_rows_1k(const double *X, int64_t ld_r, int64_t ld_k, int64_t nrows, int K, int64_t rows_p, int Kp, int RT,
                  unsigned char *planes, unsigned char *exps, cudaStream_t st, const char *who) {
  split_rows_1k_kernel<D><<<(unsigned)((rows_p / 8 + 3) / 4), 128, 0, st>>>(X, ld_r, ld_k, nrows, K, rows_p, Kp, RT,
                                                                            planes, reinterpret_cast<int *>(exps));
  return launch_status(who);
}

template <class D = Digits9x6>
int split_rows(const double *X, int64_t ld_r, int64_t ld_k, int64_t nrows, int K, int64_t rows_p, int Kp, int RT,
               unsigned char *planes, unsigned char *exps, cudaStream_t st, const char *who) {
  row_exps_kernel<<<(unsigned)((rows_p + 3) / 4), 128, 0, st>>>(X, ld_r, ld_k, nrows, K, rows_p,
                                                                 reinterpret_cast<int *>(exps));
  int rc = launch_status(who);
  if (rc) return rc;
  const int64_t warps = rows_p / 8 * ((Kp + kSplitK - 1) / kSplitK);
  split_rows_kernel<D><<<(unsigned)((warps + 3) / 4), 128, 0, st>>>(X, ld_r, ld_k, nrows, K, rows_p, Kp, RT, planes,
                                                                 reinterpret_cast<const int *>(exps));
  return launch_status(who);
}
}  // namespace tc
}  // namespace
}  // namespace dpc
