// Backward of the fused forward: from dT_i = dE/dT_i,
//   dE/dR~_ij[k] = (1/N_c) sum_m dT_i[k][m] g_m(s_ij)
//   dE/ds_ij     = (1/N_c) sum_m (sum_k dT_i[k][m] R~_ij[k]) g'_m(s_ij)
// for valid rows, zero on padding rows (Sec. II: the compressed model serves
// the backward propagation that yields forces and virials).
//
// GB300 design.  Every output of this pass belongs to one neighbour row, so
// the threads run over neighbour rows instead of channels: thread = one valid
// row, looping over the M1 channels.  Nothing is reduced across lanes -- a
// channel-parallel mapping would need five cross-lane sums per neighbour,
// each one a full-price FP64 warp instruction per shuffle level.  Per
// channel a thread evaluates g and g' together by Horner's rule (9 FMA),
// forms r_m = sum_k dT[k][m] R~[k] (4), and accumulates ds (1) and dR~ (4):
// 18 FP64 operations, all useful.  The FP64 pipe charges an instruction the
// same with 10 or 32 active lanes, so the valid rows of kGradChunk
// consecutive atoms (all type segments) are packed into one flat list and
// only the chunk's last warp can idle, instead of every atom's last warp.
// Each thread gathers its own interval's coefficients, which walk three
// contiguous planes as m advances; dT_i is read through the read-only cache
// (every lane of an atom reads the same address).  Threads past the valid
// rows zero-fill the padding rows, packed the same way.
#include <type_traits>
#include <utility>

#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kGradThreads = 128;
constexpr int kGradChunk = 16;  // atoms whose valid rows are packed together

template <typename real>
struct GradParams {
  const real *__restrict__ table;
  const io_t<real> *__restrict__ s;
  const io_t<real> *__restrict__ Rt;
  const int32_t *__restrict__ nvalid;
  const int32_t *__restrict__ atype;
  const io_t<real> *__restrict__ dT;
  io_t<real> *__restrict__ ds;
  io_t<real> *__restrict__ dRt;
  TableGeom geom;
  typename GeomOf<real>::type lgeom;  // the same geometry in the precision of real (moment kernel)
  int64_t nloc;
  int32_t nnei, ntypes, M1, pair_stride;
  int32_t sel[DP_MAX_TYPES];
  real inv_nnei;
};

// grid: x = chunk of kGradChunk atoms, y = slice of kGradThreads packed rows of that chunk
template <typename real>
__global__ void __launch_bounds__(kGradThreads) grad_kernel(const GradParams<real> P) {
  __shared__ int s_nvb[kGradChunk][DP_MAX_TYPES];
  __shared__ int s_vpre[kGradChunk + 1];  // valid rows of the chunk's atoms before atom a
  __shared__ int s_ppre[kGradChunk + 1];  // padding rows before atom a
  const int64_t a0 = (int64_t)blockIdx.x * kGradChunk;
  const int na = (int)min((int64_t)kGradChunk, P.nloc - a0);

  if (threadIdx.x < 32) {  // warp 0: counts and their prefix sums over the chunk
    const int a = threadIdx.x;
    int nv = 0;
#pragma unroll
    for (int q = 0; q < DP_MAX_TYPES; ++q) {
      int x = 0;
      if (a < na && q < P.ntypes)
        x = clampi(P.nvalid ? __ldg(P.nvalid + (a0 + a) * P.ntypes + q) : P.sel[q], 0, P.sel[q]);
      if (a < kGradChunk) s_nvb[a][q] = x;
      nv += x;
    }
    int vin = nv, pin = a < na ? P.nnei - nv : 0;  // inclusive scans
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int vu = __shfl_up_sync(0xffffffffu, vin, d), pu = __shfl_up_sync(0xffffffffu, pin, d);
      if (a >= d) {
        vin += vu;
        pin += pu;
      }
    }
    if (a < kGradChunk) {
      s_vpre[a + 1] = vin;
      s_ppre[a + 1] = pin;
    }
    if (a == 0) s_vpre[0] = s_ppre[0] = 0;
  }
  __syncthreads();

  const int v = blockIdx.y * kGradThreads + threadIdx.x;  // packed row index within the chunk
  const int nv_tot = s_vpre[kGradChunk];
  if (v < nv_tot) {
    int a = 0;
#pragma unroll
    for (int q = 1; q < kGradChunk; ++q)
      if (v >= s_vpre[q]) a = q;
    const int vv = v - s_vpre[a];
    int b = 0, cum = 0, lim = s_nvb[a][0], off = 0;
#pragma unroll
    for (int q = 1; q < DP_MAX_TYPES; ++q)
      if (q < P.ntypes && vv >= lim) {
        b = q;
        cum = lim;
        lim += s_nvb[a][q];
        off += P.sel[q - 1];
      }
    const int64_t i = a0 + a;
    const int row = off + (vv - cum);
    const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
    const Vec4<real> rr = ld4(P.Rt + (i * P.nnei + row) * 4);
    double td;
    bool clamped;
    const int l = locate(P.geom, (double)__ldg(P.s + i * P.nnei + row), td, clamped);
    const real t = (real)td;
    const real *__restrict__ cp =
        P.table + (size_t)(alpha * P.ntypes + b) * P.pair_stride + (size_t)l * P.M1 * 6;
    const real *__restrict__ dTi = P.dT + i * 4 * P.M1;
    real a_ds = real(0), a_0 = real(0), a_1 = real(0), a_2 = real(0), a_3 = real(0);
#pragma unroll 2
    for (int m = 0; m < P.M1; ++m) {
      real cf[6];
      ld6(cp, P.M1, m, cf);
      const real d0 = __ldg(dTi + m), d1 = __ldg(dTi + P.M1 + m), d2 = __ldg(dTi + 2 * P.M1 + m),
                 d3 = __ldg(dTi + 3 * P.M1 + m);
      // g and g' by Horner's rule with derivative
      real p = fma(cf[0], t, cf[1]);
      real dp = cf[0];
      dp = fma(dp, t, p);
      p = fma(p, t, cf[2]);
      dp = fma(dp, t, p);
      p = fma(p, t, cf[3]);
      dp = fma(dp, t, p);
      p = fma(p, t, cf[4]);
      dp = fma(dp, t, p);
      p = fma(p, t, cf[5]);
      real rm = d0 * rr.x;
      rm = fma(d1, rr.y, rm);
      rm = fma(d2, rr.z, rm);
      rm = fma(d3, rr.w, rm);
      a_ds = fma(rm, dp, a_ds);
      a_0 = fma(d0, p, a_0);
      a_1 = fma(d1, p, a_1);
      a_2 = fma(d2, p, a_2);
      a_3 = fma(d3, p, a_3);
    }
    if (clamped) a_ds = real(0);
    P.ds[i * P.nnei + row] = a_ds * P.inv_nnei;
    st4(P.dRt + (i * P.nnei + row) * 4, a_0 * P.inv_nnei, a_1 * P.inv_nnei, a_2 * P.inv_nnei, a_3 * P.inv_nnei);
  } else if (v - nv_tot < s_ppre[kGradChunk]) {
    // padding row number pv of the chunk, packed over atoms and their segments' padded tails
    const int pv = v - nv_tot;
    int a = 0;
#pragma unroll
    for (int q = 1; q < kGradChunk; ++q)
      if (pv >= s_ppre[q]) a = q;
    const int w = pv - s_ppre[a];
    int b = 0, cum = 0, lim = P.sel[0] - s_nvb[a][0], off = 0, nvb_b = s_nvb[a][0];
#pragma unroll
    for (int q = 1; q < DP_MAX_TYPES; ++q)
      if (q < P.ntypes && w >= lim) {
        b = q;
        cum = lim;
        lim += P.sel[q] - s_nvb[a][q];
        off += P.sel[q - 1];
        nvb_b = s_nvb[a][q];
      }
    (void)b;
    const int64_t i = a0 + a;
    const int row = off + nvb_b + (w - cum);
    P.ds[i * P.nnei + row] = real(0);
    st4(P.dRt + (i * P.nnei + row) * 4, real(0), real(0), real(0), real(0));
  }
}

// ------------------------------------------------------- interval moments
// The same backward regrouped per run of consecutive valid rows that share a
// table interval l (neighbours are sorted by distance inside a segment):
//   H[k][q] = sum_m dT[k][m] C_{l,m,q}                 (C_{l,m,q}: t^q coefficient)
//   dE/dR~_j[k] = (1/N_c) sum_q t_j^q H[k][q]
//   dE/ds_j     = (1/N_c) sum_k R~_j[k] sum_{q>=1} q t_j^(q-1) H[k][q]
// One warp per atom.  Rows are staged 32 at a time (one per lane) into a
// chunk of up to chunk_rows() rows and cut into runs; a run that reaches the end
// of a batch stays open for the next one.  When the chunk is full, the H of
// its runs are formed G runs at a time: lane = (run p, channel lane c) with
// C = 32/G channel lanes per run, each lane summing 24 products over the
// channels c, c + C, ... and a reduce-scatter over the C lanes finishing the
// sums.  Per run that is 24 M1/32 FMA (the sum itself) plus 24 log-steps'
// worth of DADD shared by G runs: with G = 8 the adds cost ~2 per run instead
// of 24 with one run across the warp.  Then every staged row (one per lane)
// follows from its run's H by Horner's rule with derivative (~45 FMA).  The
// H of an open run is kept for the next chunk.
//
// In f64 a single-row run is cheaper evaluated directly (18 M1 FMA over the
// channels, against 24 M1 for its H): such rows are queued and evaluated
// G = 8 rows at a time in the same lane layout, the five outputs of a row
// finished by a reduce-scatter over its C lanes.  In f32 the per-row form is
// bound by its scattered coefficient loads, and every run goes through H.
constexpr int kMomentWarps = 1;
// Rows staged per chunk and H slots per chunk.  df64 uses smaller chunks: its staging takes twice
// the bytes of f32's, and a one-warp block with 24 KB of shared memory left ~8 warps per SM, too few
// to hide the latencies of its long FP32 sequences (measured: 96 rows and 32 runs took the cu85
// backward from 0.459 to 0.427 ms and the water one from 0.757 to 0.688 ms; f64 keeps 128 rows).
constexpr int kDf64ChunkRows = 96;  // 64 measured the same to within 2 %
template <typename real>
constexpr int chunk_rows() { return is_df64<real> ? kDf64ChunkRows : 128; }
// df64: every run goes through H, and a row's four k components are evaluated in a loop.  Each
// df64 FMA is twelve instructions; the per-row path for single-row runs and the unrolled row
// evaluation made the kernel too large for the instruction cache (ncu: 2.0 cycles per issued
// instruction stalled on instruction fetch).  Without them the cu85 backward went from 0.533 to
// 0.459 ms and the water one from 1.018 to 0.758 ms, although single rows now cost 24 M1 + 40
// FMA instead of 18 M1.
constexpr int kDf64MinGradRun = 1;     // shortest run that goes through H in df64
constexpr bool kDf64RolledEval = true;  // evaluate a row's k components in a loop in df64
template <typename real>
constexpr int min_grad_run() { return is_df64<real> ? kDf64MinGradRun : sizeof(real) == 8 ? 2 : 1; }
// H slots per chunk (plus one for an open run's H), and the most runs one batch can add
template <typename real>
constexpr int chunk_runs() { return min_grad_run<real>() == 2 || is_df64<real> ? 32 : 64; }
template <typename real>
constexpr int batch_runs() { return 32 / min_grad_run<real>() + 1; }

template <typename real>
struct alignas(16) MomentGradStage {
  real r[chunk_rows<real>()][4];  // R~ rows of the chunk
  real t[chunk_rows<real>()];     // local variable t
  real H[chunk_runs<real>() + 1][25];  // H[run][6*k + q]; rows padded to 25 so that lanes reading different runs hit different banks
  int32_t qoff[64];  // queue of single-row runs: interval block offset and row (t and R~ are read again)
  int32_t qrow[64];
  int32_t off[chunk_rows<real>()];   // interval block offset of each staged row
  int32_t row[chunk_rows<real>()];   // row index, bit 30 set when s was clamped
  int32_t slot[chunk_rows<real>()];  // H slot of the row's run, -1 for queued rows
  int32_t run_off[chunk_runs<real>() + 1];  // interval block offset of each H slot
  int32_t nvb[DP_MAX_TYPES];
};

__host__ __device__ constexpr int ilog2(int c) { return c > 1 ? 1 + ilog2(c / 2) : 0; }

// Values a lane holds after `step` halvings of n values (an odd count is
// padded with a zero before it is halved; a single value is not split).
__host__ __device__ constexpr int rs_count(int n, int step) {
  for (int k = 0; k < step; ++k)
    if (n > 1) n = (n + 1) / 2;
  return n;
}

// Reduce-scatter of N partial sums over groups of C lanes (C a power of two,
// groups aligned to C): each step halves the values a lane holds and adds the
// partner lane's other half; once a lane holds one value the remaining steps
// add it to the partner's and the lower lane keeps it.  On return the lane
// holds the group's totals of components base .. base + nreal - 1 in
// h[0 .. nreal-1]; h needs room for N + 1 values (the padding zero).
template <int n, int mask, typename real>
__device__ __forceinline__ void rs_step(real *h, int lane, int &base, int &nreal) {
  if constexpr (mask >= 1) {
    const bool hi = lane & mask;
    if constexpr (n == 1) {
      h[0] += shfl_xor(h[0], mask);
      if (hi) nreal = 0;
      rs_step<1, mask / 2>(h, lane, base, nreal);
    } else {
      if constexpr ((n & 1) != 0) h[n] = real(0);
      constexpr int half = (n + 1) / 2;
#pragma unroll
      for (int x = 0; x < half; ++x) {
        const real snd = hi ? h[x] : h[x + half], kp = hi ? h[x + half] : h[x];
        h[x] = kp + shfl_xor(snd, mask);
      }
      if (hi) {
        base += half;
        nreal = max(nreal - half, 0);
      } else {
        nreal = min(nreal, half);
      }
      rs_step<half, mask / 2>(h, lane, base, nreal);
    }
  }
}

template <int N, int C, typename real>
__device__ __forceinline__ void reduce_scatter(real *h, int lane, int &base, int &nreal) {
  base = 0;
  nreal = N;
  rs_step<N, C / 2>(h, lane, base, nreal);
}

// Channel loops are unrolled twice in f64 and f32.  In df64 every FMA is
// twelve instructions: the loop bodies are large already, and a kernel that
// no longer fits the instruction cache stalls on instruction fetch.
template <typename real>
constexpr int kUnrollM = is_df64<real> ? 1 : 2;

// H of the runs in slots s0 .. s0+G-1 (those below nrun): lane = (run p, channel lane c),
// C = 32/G channel lanes per run, each summing over the channels c, c + C, ...
template <int G, typename real>
__device__ __forceinline__ void form_H_group(MomentGradStage<real> &st, const real *__restrict__ tab,
                                             const real *dts, int M1, int s0, int nrun, int lane) {
  constexpr int C = 32 / G;
  const int p = lane / C, c = lane - p * C;
  const int slot = s0 + p;
  const bool valid = slot < nrun;
  const real *__restrict__ blk = tab + st.run_off[valid ? slot : s0];
  real h[25];
#pragma unroll
  for (int x = 0; x < 24; ++x) h[x] = real(0);
#pragma unroll kUnrollM<real>
  for (int m = c; m < M1; m += C) {
    real c6[6];  // (a..f): coefficients of t^5 .. t^0
    ld6(blk, M1, m, c6);
    const real d0 = dts[m * 4 + 0], d1 = dts[m * 4 + 1], d2 = dts[m * 4 + 2], d3 = dts[m * 4 + 3];
#pragma unroll
    for (int q = 0; q < 6; ++q) {
      h[0 * 6 + q] = fma(d0, c6[5 - q], h[0 * 6 + q]);
      h[1 * 6 + q] = fma(d1, c6[5 - q], h[1 * 6 + q]);
      h[2 * 6 + q] = fma(d2, c6[5 - q], h[2 * 6 + q]);
      h[3 * 6 + q] = fma(d3, c6[5 - q], h[3 * 6 + q]);
    }
  }
  int base, nreal;
  reduce_scatter<24, C>(h, lane, base, nreal);
  if (valid) {
#pragma unroll
    for (int x = 0; x < rs_count(24, ilog2(C)); ++x)
      if (x < nreal) st.H[slot][base + x] = h[x];
  }
}

// Per-row backward of queued rows q0 .. q0+G-1 (those below nq): lane = (row p, channel lane c),
// each lane summing the five outputs over the channels c, c + C, ... (18 FMA per channel).
// dts holds dT_i / N_c, so the sums are the outputs.
template <int G, typename real>
__device__ __forceinline__ void grad_rows_group(const GradParams<real> &P, const MomentGradStage<real> &st,
                                                const real *__restrict__ tab, const real *dts, int64_t i, int q0,
                                                int nq, int lane) {
  constexpr int kClamped = 1 << 30;
  constexpr int C = 32 / G;
  const int p = lane / C, c = lane - p * C;
  const int q = q0 + p;
  const bool valid = q < nq;
  const int e = valid ? q : q0;
  const int rw = st.qrow[e];
  const int row = rw & (kClamped - 1);
  const Vec4<real> rr = ld4r<real>(P.Rt + (i * P.nnei + row) * 4);
  real t;
  bool clamped;
  locate(P.lgeom, __ldg(P.s + i * P.nnei + row), t, clamped);
  const real *__restrict__ blk = tab + st.qoff[e];
  const int M1 = P.M1;
  real a[6];  // ds, dR~[0..3], and room for the padding zero
#pragma unroll
  for (int x = 0; x < 5; ++x) a[x] = real(0);
#pragma unroll kUnrollM<real>
  for (int m = c; m < M1; m += C) {
    real cf[6];
    ld6(blk, M1, m, cf);
    const real d0 = dts[m * 4 + 0], d1 = dts[m * 4 + 1], d2 = dts[m * 4 + 2], d3 = dts[m * 4 + 3];
    real g = fma(cf[0], t, cf[1]);  // g and g' by Horner's rule with derivative
    real dg = cf[0];
    dg = fma(dg, t, g);
    g = fma(g, t, cf[2]);
    dg = fma(dg, t, g);
    g = fma(g, t, cf[3]);
    dg = fma(dg, t, g);
    g = fma(g, t, cf[4]);
    dg = fma(dg, t, g);
    g = fma(g, t, cf[5]);
    real rm = d0 * rr.x;
    rm = fma(d1, rr.y, rm);
    rm = fma(d2, rr.z, rm);
    rm = fma(d3, rr.w, rm);
    a[0] = fma(rm, dg, a[0]);
    a[1] = fma(d0, g, a[1]);
    a[2] = fma(d1, g, a[2]);
    a[3] = fma(d2, g, a[3]);
    a[4] = fma(d3, g, a[4]);
  }
  int base, nreal;
  reduce_scatter<5, C>(a, lane, base, nreal);
  if (valid) {
    io_t<real> *__restrict__ ds_i = P.ds + i * P.nnei;
    io_t<real> *__restrict__ dR_i = P.dRt + i * P.nnei * 4;
#pragma unroll
    for (int x = 0; x < rs_count(5, ilog2(C)); ++x)
      if (x < nreal) {
        const int comp = base + x;
        if (comp == 0)
          ds_i[row] = (rw & kClamped) ? io_t<real>(0) : to_io(a[x]);
        else
          dR_i[(size_t)row * 4 + comp - 1] = to_io(a[x]);
      }
  }
}

// Group size for `rem` runs or rows left: G = 8 for 7 or more, then 4, 2, 1.  df64 keeps two
// of the four shapes (8 for 5 or more, else 1): each shape is another copy of a large loop.
template <typename real>
__device__ __forceinline__ int h_group_size(int rem) {
  if constexpr (is_df64<real>) return rem >= 5 ? 8 : 1;
  return rem >= 7 ? 8 : rem >= 4 ? 4 : rem >= 2 ? 2 : 1;
}

template <typename real>
__device__ __forceinline__ void form_H_runs(MomentGradStage<real> &st, const real *__restrict__ tab, const real *dts,
                                            int M1, int nrun, int lane) {
  for (int s0 = 0; s0 < nrun;) {  // uniform
    const int G = h_group_size<real>(nrun - s0);
    if constexpr (is_df64<real>) {
      if (G == 8)
        form_H_group<8>(st, tab, dts, M1, s0, nrun, lane);
      else
        form_H_group<1>(st, tab, dts, M1, s0, nrun, lane);
      s0 += G;
      continue;
    }
    if (G == 8)
      form_H_group<8>(st, tab, dts, M1, s0, nrun, lane);
    else if (G == 4)
      form_H_group<4>(st, tab, dts, M1, s0, nrun, lane);
    else if (G == 2)
      form_H_group<2>(st, tab, dts, M1, s0, nrun, lane);
    else
      form_H_group<1>(st, tab, dts, M1, s0, nrun, lane);
    s0 += G;
  }
}

// Queued rows q0 .. n-1 in groups: G = 8 while `all` is false (the rest stays queued), else down to 1.
template <typename real>
__device__ __forceinline__ int grad_rows_queued(const GradParams<real> &P, const MomentGradStage<real> &st,
                                                const real *__restrict__ tab, const real *dts, int64_t i, int n,
                                                bool all, int lane) {
  int q0 = 0;
  while (n - q0 >= 8 || (all && q0 < n)) {  // uniform
    const int G = h_group_size<real>(n - q0);
    if constexpr (is_df64<real>) {
      if (G == 8)
        grad_rows_group<8>(P, st, tab, dts, i, q0, n, lane);
      else
        grad_rows_group<1>(P, st, tab, dts, i, q0, n, lane);
      q0 += G;
      continue;
    }
    if (G == 8)
      grad_rows_group<8>(P, st, tab, dts, i, q0, n, lane);
    else if (G == 4)
      grad_rows_group<4>(P, st, tab, dts, i, q0, n, lane);
    else if (G == 2)
      grad_rows_group<2>(P, st, tab, dts, i, q0, n, lane);
    else
      grad_rows_group<1>(P, st, tab, dts, i, q0, n, lane);
    q0 += G;
  }
  return q0;
}

template <typename real>
__global__ void __launch_bounds__(kMomentWarps * 32) grad_moments_kernel(const GradParams<real> P) {
  constexpr int kClamped = 1 << 30;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int lane = threadIdx.x & 31;
  const int64_t i = blockIdx.x;  // one atom per block (one warp)
  MomentGradStage<real> &st = *reinterpret_cast<MomentGradStage<real> *>(smem_raw);
  real *dts = reinterpret_cast<real *>(smem_raw + sizeof(MomentGradStage<real>));  // [M1][4]
  const int M1 = P.M1;

  {  // counts in shared memory
    int sl = 0;
#pragma unroll
    for (int q = 0; q < DP_MAX_TYPES; ++q)
      if (lane == q) sl = P.sel[q];
    int x = 0;
    if (lane < P.ntypes) x = clampi(P.nvalid ? __ldg(P.nvalid + i * P.ntypes + lane) : sl, 0, sl);
    if (lane < DP_MAX_TYPES) st.nvb[lane] = x;
  }
  {  // dT_i / N_c, transposed: the 1/N_c of every output is folded in here, once per atom
    const io_t<real> *__restrict__ dTi = P.dT + i * 4 * M1;
#pragma unroll 4
    for (int e = lane; e < 4 * M1; e += 32) {  // unrolled: several loads in flight per lane
      const int k = e / M1, m = e - k * M1;
      dts[m * 4 + k] = from_io<real>(__ldg(dTi + e)) * P.inv_nnei;
    }
  }
  __syncwarp();
  int nv = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q) nv += st.nvb[q];
  const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
  const real *__restrict__ tab = P.table + (size_t)alpha * P.ntypes * P.pair_stride;
  io_t<real> *__restrict__ ds_i = P.ds + i * P.nnei;
  io_t<real> *__restrict__ dR_i = P.dRt + i * P.nnei * 4;

  // outputs of one row (this lane) from its run's H, by Horner's rule with derivative
  auto eval_row = [&](const real *Hr, real t, real r0, real r1, real r2, real r3, int rw) {
    const int row = rw & (kClamped - 1);
    real dsv = real(0);
    if constexpr (is_df64<real> && kDf64RolledEval) {
      // one k component per iteration: a quarter of the code, each output stored as it is done
#pragma unroll 1
      for (int k = 0; k < 4; ++k) {
        const real *hk = Hr + 6 * k;
        real p = fma(hk[5], t, hk[4]);
        real dp = hk[5];
        dp = fma(dp, t, p);
        p = fma(p, t, hk[3]);
        dp = fma(dp, t, p);
        p = fma(p, t, hk[2]);
        dp = fma(dp, t, p);
        p = fma(p, t, hk[1]);
        dp = fma(dp, t, p);
        p = fma(p, t, hk[0]);
        const real rk = k == 0 ? r0 : k == 1 ? r1 : k == 2 ? r2 : r3;
        dsv = fma(rk, dp, dsv);
        dR_i[(size_t)row * 4 + k] = to_io(p);
      }
    } else {
      real dR[4], G[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const real *hk = Hr + 6 * k;  // H[k][q], q = 0..5
        real p = fma(hk[5], t, hk[4]);
        real dp = hk[5];
        dp = fma(dp, t, p);
        p = fma(p, t, hk[3]);
        dp = fma(dp, t, p);
        p = fma(p, t, hk[2]);
        dp = fma(dp, t, p);
        p = fma(p, t, hk[1]);
        dp = fma(dp, t, p);
        p = fma(p, t, hk[0]);
        dR[k] = p;
        G[k] = dp;
      }
      dsv = r0 * G[0];
      dsv = fma(r1, G[1], dsv);
      dsv = fma(r2, G[2], dsv);
      dsv = fma(r3, G[3], dsv);
      st4(dR_i + (size_t)row * 4, dR[0], dR[1], dR[2], dR[3]);
    }
    ds_i[row] = (rw & kClamped) ? io_t<real>(0) : to_io(dsv);
  };
  constexpr int kCarrySlot = chunk_runs<real>();

  int nrows = 0, nrun = 0;  // staged rows and runs of the chunk (uniform)
  int nq = 0;               // queued rows (uniform)
  int last_off = -1, last_slot = -1;
  bool last_open = false;   // the last run may go on in the next batch
  for (int base = 0; base < nv; base += 32) {
    const int cnt = min(32, nv - base);
    if (lane < cnt) {  // stage row base + lane at chunk position nrows + lane
      const int v = base + lane;
      int b = 0, cum = 0, lim = st.nvb[0], off = 0;
#pragma unroll
      for (int c = 1; c < DP_MAX_TYPES; ++c)
        if (c < P.ntypes && v >= lim) {
          b = c;
          cum = lim;
          lim += st.nvb[c];
          off += P.sel[c - 1];
        }
      const int row = off + (v - cum);
      const Vec4<real> rr = ld4r<real>(P.Rt + (i * P.nnei + row) * 4);
      real t;
      bool clamped;
      const int l = locate(P.lgeom, __ldg(P.s + i * P.nnei + row), t, clamped);
      const int j = nrows + lane;
      st.r[j][0] = rr.x;
      st.r[j][1] = rr.y;
      st.r[j][2] = rr.z;
      st.r[j][3] = rr.w;
      st.t[j] = t;
      st.off[j] = (b * P.geom.nint + l) * M1 * 6;
      st.row[j] = row | (clamped ? kClamped : 0);
    }
    __syncwarp();
    const bool more = base + cnt < nv;
    // run starts of the batch: rows whose interval block differs from the previous row's
    const int myoff = lane < cnt ? st.off[nrows + lane] : -1;
    const int prevoff = __shfl_up_sync(0xffffffffu, myoff, 1);
    unsigned starts = __ballot_sync(0xffffffffu, lane < cnt && (lane == 0 || myoff != prevoff));
    while (starts) {  // uniform, run by run
      const int u = __ffs(starts) - 1;
      starts &= starts - 1;
      const int e = starts ? __ffs(starts) - 1 : cnt;
      const int off = __shfl_sync(0xffffffffu, myoff, u);
      int slot;
      if (u == 0 && last_open && off == last_off) {
        slot = last_slot;  // the previous batch's last run goes on
      } else if (e - u >= min_grad_run<real>() || (e == cnt && more)) {
        slot = nrun++;
        if (lane == 0) st.run_off[slot] = off;
      } else {
        slot = -1;  // a single-row run: queue it
        if (lane == 0) {
          st.qoff[nq] = off;
          st.qrow[nq] = st.row[nrows + u];
        }
        ++nq;
      }
      if (lane >= u && lane < e) st.slot[nrows + lane] = slot;
      if (e == cnt) {
        last_off = off;
        last_slot = slot;
        last_open = more && slot >= 0;
      }
    }
    nrows += cnt;
    __syncwarp();
    if (nrows + 32 > chunk_rows<real>() || nrun + batch_runs<real>() > chunk_runs<real>() || !more) {  // chunk full, or the atom's last rows
      form_H_runs(st, tab, dts, M1, nrun, lane);
      __syncwarp();
      for (int j = lane; j < nrows; j += 32) {
        const int sl = st.slot[j];
        if (sl >= 0) eval_row(st.H[sl], st.t[j], st.r[j][0], st.r[j][1], st.r[j][2], st.r[j][3], st.row[j]);
      }
      __syncwarp();
      if (last_open && last_slot != kCarrySlot) {  // keep the open run's H for the next chunk
        if (lane < 24) st.H[kCarrySlot][lane] = st.H[last_slot][lane];
        last_slot = kCarrySlot;
      }
      nrows = 0;
      nrun = 0;
      __syncwarp();
    }
    if (min_grad_run<real>() > 1 && nq >= 8) {  // single-row runs, 8 at a time; fewer than 8 stay queued
      const int done = grad_rows_queued(P, st, tab, dts, i, nq, false, lane);
      __syncwarp();
      if (lane < nq - done) {
        st.qoff[lane] = st.qoff[done + lane];
        st.qrow[lane] = st.qrow[done + lane];
      }
      nq -= done;
      __syncwarp();
    }
  }
  if constexpr (min_grad_run<real>() > 1) grad_rows_queued(P, st, tab, dts, i, nq, true, lane);

  // padding rows, packed over the segments' padded tails
  for (int pv = lane; pv < P.nnei - nv; pv += 32) {
    int cum = 0, lim = P.sel[0] - st.nvb[0], off = 0, nvb_b = st.nvb[0];
#pragma unroll
    for (int c = 1; c < DP_MAX_TYPES; ++c)
      if (c < P.ntypes && pv >= lim) {
        cum = lim;
        lim += P.sel[c] - st.nvb[c];
        off += P.sel[c - 1];
        nvb_b = st.nvb[c];
      }
    const int row = off + nvb_b + (pv - cum);
    ds_i[row] = io_t<real>(0);
    st4(dR_i + (size_t)row * 4, io_t<real>(0), io_t<real>(0), io_t<real>(0), io_t<real>(0));
  }
}

// ---------------------------------------------------------------- f32
// In f32 the FFMA pipe is 64x faster than FP64 and the per-thread gather of
// a private coefficient row (32 distinct lines per load instruction) would
// bind long before the arithmetic.  So the f32 backward works on row groups:
// L channel lanes per neighbour row and 32/L rows per warp instruction.  The
// L lanes of a row read L consecutive channels of the row's interval (three
// contiguous runs of 8*L bytes in the pair-planar block), and rows that share
// an interval -- most neighbours next to each other in distance order -- hit
// the same sectors.  Each warp prepares 32 rows at a time (segment lookup,
// interval search, R~ load) spread over its lanes, and the row groups read
// them back as shared-memory broadcasts.  dT_i sits in shared memory as
// [M1][4] (one 16-byte load per channel round), which keeps the register
// count low enough for the occupancy that hides the coefficient loads.  The
// five per-row sums (ds, dR~[0..3]) meet in a log2(L)-level shuffle
// reduction per row, amortised over the M1/L channel rounds of that row.
constexpr int kGradF32Warps = 4;

struct GradParamsF32 {
  const float *__restrict__ table;
  const float *__restrict__ s;
  const float *__restrict__ Rt;
  const int32_t *__restrict__ nvalid;
  const int32_t *__restrict__ atype;
  const float *__restrict__ dT;
  float *__restrict__ ds;
  float *__restrict__ dRt;
  TableGeomF geom;
  int64_t nloc;
  int32_t nnei, ntypes, M1, pair_stride;
  int32_t sel[DP_MAX_TYPES];
  float inv_nnei;
};

// Per-warp staging of 32 valid rows: prepared once per row, lane-distributed,
// then read by the row groups as shared-memory broadcasts.
struct alignas(16) RowStage {
  float4 r[32];     // R~ rows
  float t[32];      // local variable t
  int32_t blk[32];  // element offset of the interval's coefficient block (centre type's tables)
  int32_t row[32];  // row index, with bit 30 set when s was clamped (ds = 0)
};

template <int L, int R>
__global__ void __launch_bounds__(kGradF32Warps * 32) grad_f32_kernel(const GradParamsF32 P) {
  constexpr int RPW = 32 / L;  // rows per warp instruction
  constexpr int kClamped = 1 << 30;
  __shared__ RowStage stage[kGradF32Warps];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int grp = lane / L, q = lane % L;
  const int64_t i = blockIdx.x;  // one atom per block
  RowStage &st = stage[w];

  int nvb[DP_MAX_TYPES];
  int nv = 0;
#pragma unroll
  for (int b = 0; b < DP_MAX_TYPES; ++b) {
    int x = 0;
    if (b < P.ntypes) x = clampi(P.nvalid ? __ldg(P.nvalid + i * P.ntypes + b) : P.sel[b], 0, P.sel[b]);
    nvb[b] = x;
    nv += x;
  }
  const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
  const float *__restrict__ tab = P.table + (size_t)alpha * P.ntypes * P.pair_stride;
  float *__restrict__ ds_i = P.ds + i * P.nnei;
  float *__restrict__ dR_i = P.dRt + i * P.nnei * 4;

  // dT_i transposed to [L*R][4] in shared memory (zero past M1): one 16-byte load per channel round
  __shared__ float4 dts[L * R];
  {
    const float *__restrict__ dTi = P.dT + i * 4 * P.M1;
    for (int m = threadIdx.x; m < L * R; m += kGradF32Warps * 32)
      dts[m] = m < P.M1 ? make_float4(__ldg(dTi + m), __ldg(dTi + P.M1 + m), __ldg(dTi + 2 * P.M1 + m),
                                      __ldg(dTi + 3 * P.M1 + m))
                        : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  }
  __syncthreads();

  for (int base = 32 * w; base < nv; base += 32 * kGradF32Warps) {  // warp-uniform
    const int cnt = min(32, nv - base);
    if (lane < cnt) {  // stage row base + lane
      const int v = base + lane;
      int b = 0, cum = 0, lim = nvb[0], off = 0;
#pragma unroll
      for (int c = 1; c < DP_MAX_TYPES; ++c)
        if (c < P.ntypes && v >= lim) {
          b = c;
          cum = lim;
          lim += nvb[c];
          off += P.sel[c - 1];
        }
      const int row = off + (v - cum);
      const Vec4<float> rr = ld4(P.Rt + (i * P.nnei + row) * 4);
      float t;
      bool clamped;
      const int l = locate(P.geom, __ldg(P.s + i * P.nnei + row), t, clamped);
      st.r[lane] = make_float4(rr.x, rr.y, rr.z, rr.w);
      st.t[lane] = t;
      st.blk[lane] = (b * P.geom.nint + l) * P.M1 * 6;
      st.row[lane] = row | (clamped ? kClamped : 0);
    }
    __syncwarp();
    for (int u0 = 0; u0 < cnt; u0 += RPW) {  // warp-uniform
      const int u = u0 + grp;
      const bool act = u < cnt;
      float a_ds = 0.0f, a_0 = 0.0f, a_1 = 0.0f, a_2 = 0.0f, a_3 = 0.0f;
      if (act) {
        const float4 rr = st.r[u];
        const float t = st.t[u];
        const float2 *q0 = reinterpret_cast<const float2 *>(tab + st.blk[u]) + q;
        const float2 *q1 = q0 + P.M1, *q2 = q1 + P.M1;
#pragma unroll
        for (int r = 0; r < R; ++r) {
          if (r < R - 1 || q + L * r < P.M1) {
            const float2 ab = __ldg(q0 + L * r), cd = __ldg(q1 + L * r), ef = __ldg(q2 + L * r);
            const float4 d = dts[q + L * r];
            float p = fmaf(ab.x, t, ab.y);
            float dp = ab.x;
            dp = fmaf(dp, t, p);
            p = fmaf(p, t, cd.x);
            dp = fmaf(dp, t, p);
            p = fmaf(p, t, cd.y);
            dp = fmaf(dp, t, p);
            p = fmaf(p, t, ef.x);
            dp = fmaf(dp, t, p);
            p = fmaf(p, t, ef.y);
            float rm = d.x * rr.x;
            rm = fmaf(d.y, rr.y, rm);
            rm = fmaf(d.z, rr.z, rm);
            rm = fmaf(d.w, rr.w, rm);
            a_ds = fmaf(rm, dp, a_ds);
            a_0 = fmaf(d.x, p, a_0);
            a_1 = fmaf(d.y, p, a_1);
            a_2 = fmaf(d.z, p, a_2);
            a_3 = fmaf(d.w, p, a_3);
          }
        }
      }
#pragma unroll
      for (int sh = L / 2; sh > 0; sh >>= 1) {
        a_ds += __shfl_xor_sync(0xffffffffu, a_ds, sh);
        a_0 += __shfl_xor_sync(0xffffffffu, a_0, sh);
        a_1 += __shfl_xor_sync(0xffffffffu, a_1, sh);
        a_2 += __shfl_xor_sync(0xffffffffu, a_2, sh);
        a_3 += __shfl_xor_sync(0xffffffffu, a_3, sh);
      }
      if (act && q == 0) {
        const int rw = st.row[u];
        const int row = rw & (kClamped - 1);
        ds_i[row] = (rw & kClamped) ? 0.0f : a_ds * P.inv_nnei;
        st4(dR_i + (size_t)row * 4, a_0 * P.inv_nnei, a_1 * P.inv_nnei, a_2 * P.inv_nnei, a_3 * P.inv_nnei);
      }
    }
    __syncwarp();
  }

  // padding rows of this atom, packed over the segments' padded tails
  for (int pv = threadIdx.x; pv < P.nnei - nv; pv += kGradF32Warps * 32) {
    int cum = 0, lim = P.sel[0] - nvb[0], off = 0, nvb_b = nvb[0];
#pragma unroll
    for (int c = 1; c < DP_MAX_TYPES; ++c)
      if (c < P.ntypes && pv >= lim) {
        cum = lim;
        lim += P.sel[c] - nvb[c];
        off += P.sel[c - 1];
        nvb_b = nvb[c];
      }
    const int row = off + nvb_b + (pv - cum);
    ds_i[row] = 0.0f;
    st4(dR_i + (size_t)row * 4, 0.0f, 0.0f, 0.0f, 0.0f);
  }
}

using GradF32Kernel = void (*)(const GradParamsF32);

template <int L, int... Rs>
GradF32Kernel pick_grad_f32(int R, std::integer_sequence<int, Rs...>) {
  GradF32Kernel k = nullptr;
  ((R == Rs + 1 ? (k = &grad_f32_kernel<L, Rs + 1>, 0) : 0), ...);
  return k;
}

int grad_f32(const float *table, const TableGeom &g, const Segments &seg, const float *s, const float *Rt,
             const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes, int M1, const float *dT,
             float *ds, float *dRt, void *stream) {
  GradParamsF32 P;
  P.table = table;
  P.s = s;
  P.Rt = Rt;
  P.nvalid = nvalid;
  P.atype = atype;
  P.dT = dT;
  P.ds = ds;
  P.dRt = dRt;
  P.geom = to_f32(g);
  P.nloc = nloc;
  P.nnei = nnei;
  P.ntypes = ntypes;
  P.M1 = M1;
  P.pair_stride = g.nint * M1 * 6;
  for (int b = 0; b < DP_MAX_TYPES; ++b) P.sel[b] = seg.sel[b];
  P.inv_nnei = (float)(1.0 / (double)nnei);
  // 8 channel lanes per row up to M1 = 128 (at most 16 rounds), 16 beyond
  const int L = M1 <= 128 ? 8 : 16;
  const int R = (M1 + L - 1) / L;
  GradF32Kernel k = L == 8 ? pick_grad_f32<8>(R, std::make_integer_sequence<int, 16>{})
                           : pick_grad_f32<16>(R, std::make_integer_sequence<int, 16>{});
  if (!k) return set_error(DP_ERR_UNSUPPORTED, "no f32 gradient kernel for M1 = %d", M1);
  k<<<(unsigned)nloc, kGradF32Warps * 32, 0, (cudaStream_t)stream>>>(P);
  return launch_status("dp_tabulate_fusion_grad_f32");
}

template <typename real>
int grad(const real *table, const dp_table_info *info, const io_t<real> *s, const io_t<real> *Rt,
         const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1,
         const io_t<real> *dT, io_t<real> *ds, io_t<real> *dRt, void *stream, bool moments = false) {
  clear_error();
  TableGeom g;
  Segments seg;
  int rc = check_fusion_args(table, info, s, Rt, nloc, nnei, ntypes, sel, M1, ds, dRt, &g, &seg);
  if (rc) return rc;
  if (nloc == 0) return DP_OK;
  if (!dT) return set_error(DP_ERR_NULL, "dT is NULL");
  if (nloc > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
  if constexpr (std::is_same<real, float>::value)
    if (!moments) return grad_f32(table, g, seg, s, Rt, nvalid, atype, nloc, nnei, ntypes, M1, dT, ds, dRt, stream);
  GradParams<real> P;
  P.table = table;
  P.s = s;
  P.Rt = Rt;
  P.nvalid = nvalid;
  P.atype = atype;
  P.dT = dT;
  P.ds = ds;
  P.dRt = dRt;
  P.geom = g;
  P.lgeom = GeomOf<real>::make(g);
  P.nloc = nloc;
  P.nnei = nnei;
  P.ntypes = ntypes;
  P.M1 = M1;
  P.pair_stride = g.nint * M1 * 6;
  for (int b = 0; b < DP_MAX_TYPES; ++b) P.sel[b] = seg.sel[b];
  P.inv_nnei = host_cvt<real>(1.0 / (double)nnei);
  if (moments) {
    void (*k)(const GradParams<real>) = &grad_moments_kernel<real>;
    const size_t smem = sizeof(MomentGradStage<real>) + (size_t)4 * M1 * sizeof(real);
    if (smem > 48 * 1024) {
      const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_tabulate_fusion_grad_moments: %s", cudaGetErrorString(e));
    }
    k<<<(unsigned)nloc, kMomentWarps * 32, smem, (cudaStream_t)stream>>>(P);
    return launch_status("dp_tabulate_fusion_grad_moments");
  }
  if constexpr (std::is_same<real, df64>::value) {
    return set_error(DP_ERR_UNSUPPORTED, "df64 runs the moment form only");
  } else {
  const int64_t ychunks = ((int64_t)kGradChunk * nnei + kGradThreads - 1) / kGradThreads;
  if (ychunks > 65535) return set_error(DP_ERR_SHAPE, "nnei = %d too large", nnei);
  const int64_t xchunks = (nloc + kGradChunk - 1) / kGradChunk;
  dim3 grid((unsigned)xchunks, (unsigned)ychunks);
  grad_kernel<real><<<grid, kGradThreads, 0, (cudaStream_t)stream>>>(P);
  return launch_status("dp_tabulate_fusion_grad");
  }
}

}  // namespace

}  // namespace dpc

extern "C" {

int dp_tabulate_fusion_grad_f64(const double *table, const dp_table_info *info, const double *s, const double *Rt,
                                const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                const int32_t *sel, int M1, const double *dT, double *ds, double *dRt,
                                void *stream) {
  return dpc::grad<double>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, dT, ds, dRt, stream);
}

int dp_tabulate_fusion_grad_f32(const float *table, const dp_table_info *info, const float *s, const float *Rt,
                                const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                const int32_t *sel, int M1, const float *dT, float *ds, float *dRt, void *stream) {
  return dpc::grad<float>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, dT, ds, dRt, stream);
}

int dp_tabulate_fusion_grad_moments_f64(const double *table, const dp_table_info *info, const double *s,
                                        const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                        int nnei, int ntypes, const int32_t *sel, int M1, const double *dT, double *ds,
                                        double *dRt, void *stream) {
  return dpc::grad<double>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, dT, ds, dRt, stream, true);
}

int dp_tabulate_fusion_grad_moments_df64(const float *table, const dp_table_info *info, const double *s,
                                         const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                         int nnei, int ntypes, const int32_t *sel, int M1, const double *dT,
                                         double *ds, double *dRt, void *stream) {
  return dpc::grad<dpc::df64>(reinterpret_cast<const dpc::df64 *>(table), info, s, Rt, nvalid, atype, nloc, nnei,
                              ntypes, sel, M1, dT, ds, dRt, stream, true);
}

int dp_tabulate_fusion_grad_moments_f32(const float *table, const dp_table_info *info, const float *s,
                                        const float *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                        int nnei, int ntypes, const int32_t *sel, int M1, const float *dT, float *ds,
                                        float *dRt, void *stream) {
  return dpc::grad<float>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, dT, ds, dRt, stream, true);
}

}  // extern "C"
