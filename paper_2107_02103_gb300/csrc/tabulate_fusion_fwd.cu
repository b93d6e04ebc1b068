// Fused tabulated embedding + contraction, forward (Sec. II, kernel fusion):
//   T_i[k][m] = (1/N_c) sum over valid rows j of R~_ij[k] * g_m(s_ij)
// G_i is never stored: each row's M1 polynomial values live in registers
// only for the four FMAs that fold them into T_i.  Padded rows are skipped
// through the per-type valid counts.
//
// GB300 design.  The FP64 pipe issues one warp instruction per 16 SM clocks
// however many lanes are active, so every FP64 instruction must have 32 busy
// lanes.  With M1 = 32 Q + RR:
//   * Q full rounds: all 32 lanes work on the same neighbour, lane l owning
//     channels l, l + 32, ..., l + 32 (Q-1).  The interval's coefficients
//     are one contiguous 6*M1 block, pair-planar, so each round's three
//     vector loads are fully coalesced.
//   * one packed round for the RR remaining channels: lane l serves channel
//     32 Q + (l mod RR) of neighbour l / RR, so PK = 32 / RR neighbours share
//     one instruction (M1 = 100: 4 remainder channels x 8 neighbours fill all
//     32 lanes, so 100 channels cost exactly 100/32 instructions).
//   * the interval search, the segment lookup and the R~ row load run once
//     per neighbour, spread over the lanes (lane l handles neighbour base +
//     l), and are handed over through shared memory: their FP64 work costs
//     1/32 of an instruction per neighbour.
//   * one warp per block and per atom keeps the work units small, so the
//     block scheduler balances the SMs to within a few atoms.
// The same kernels run in df64 (double-float) arithmetic on the FP32 pipes
// for double inputs and outputs: the templates are written against the
// arithmetic type `real` and read / write arrays of io_t<real>.
// The packed round's partial sums meet in a shuffle reduction over the PK
// lanes of each remainder channel, once per atom.  In f32 the coefficient
// row of the current interval is also kept in registers across consecutive
// neighbours that share it (sorted by distance, they often do): there the
// L1 traffic of reloading it, not the FFMA pipe, would be the limit.
#include <type_traits>
#include <utility>

#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kFwdWarps = 1;

template <typename real>
struct FwdParams {
  const real *__restrict__ table;
  const io_t<real> *__restrict__ s;
  const io_t<real> *__restrict__ Rt;
  const int32_t *__restrict__ nvalid;
  const int32_t *__restrict__ atype;
  io_t<real> *__restrict__ T;
  io_t<real> *__restrict__ D;  // optional fused descriptor output [nloc][M1][M2] (NULL: T only)
  typename GeomOf<real>::type geom;
  int64_t nloc;
  int32_t nnei, ntypes, M1, pair_stride;  // pair_stride = nint * M1 * 6
  int32_t RR, PK;                          // remainder channels, neighbours per packed round
  int32_t M2;                              // descriptor width when D is set (M2 <= 32)
  int32_t sel[DP_MAX_TYPES];
  real inv_nnei;
};

template <typename real>
struct alignas(16) Stage {
  real r[32][4];    // R~ rows of the staged neighbours
  real t[32];       // local variable t
  int32_t off[32];  // element offset of the interval's coefficient block in the centre type's tables
  int32_t nvb[DP_MAX_TYPES];  // valid rows per type segment of the current atom
};

// Extra staging of the interval-moment variant: powers t^0..t^5 of every
// staged neighbour, the 24 moments W[k][q] of the last runs contracted (kept
// until the remainder channels of up to kPendRuns runs are done in one packed
// round), their interval blocks, and the rows of the batch's short runs.
constexpr int kPendRuns = 8;
template <typename real>
struct alignas(16) MomentStage {
  real tp[32][6];
  real w[kPendRuns][24];
  int32_t poff[kPendRuns];
  int32_t srow[32];
};

// Runs at least this long go through interval moments; shorter ones are
// evaluated neighbour by neighbour (a run costs n + 24 Q FMA instructions in
// moments against 9 Q n per neighbour).
constexpr int kMinMomentRun = 3;
// df64: runs of 3 rows are cheaper per row in time although not in FMA count (measured: water
// forward 0.481 -> 0.436 ms, Al-Cu-Mg 2.58 -> 2.51 ms, cu85 0.295 -> 0.298 ms with 4).
constexpr int kDf64MinMomentRun = 4;
template <typename real>
constexpr int min_moment_run() { return is_df64<real> ? kDf64MinMomentRun : kMinMomentRun; }

template <typename real>
__device__ __forceinline__ real horner5(const real c[6], real t) {
  // g = ((((a t + b) t + c) t + d) t + e) t + f
  real g = fma(c[0], t, c[1]);
  g = fma(g, t, c[2]);
  g = fma(g, t, c[3]);
  g = fma(g, t, c[4]);
  return fma(g, t, c[5]);
}

// One neighbour (interval block offset `off`, local t, R~ row r) folded into
// the lane's Q channel rounds, coefficients loaded round by round (f64).
template <typename real, int Q>
__device__ __forceinline__ void fwd_neighbour(const FwdParams<real> &P, const real *__restrict__ tab, const int lane,
                                              const int off, const real t, const real *r,
                                              real (&acc)[Q > 0 ? Q : 1][4]) {
  const real r0 = r[0], r1 = r[1], r2 = r[2], r3 = r[3];
#pragma unroll
  for (int k = 0; k < Q; ++k) {
    real c6[6];
    ld6(tab + off, P.M1, k * 32 + lane, c6);
    const real g = horner5(c6, t);
    acc[k][0] = fma(r0, g, acc[k][0]);
    acc[k][1] = fma(r1, g, acc[k][1]);
    acc[k][2] = fma(r2, g, acc[k][2]);
    acc[k][3] = fma(r3, g, acc[k][3]);
  }
}

// f32: the coefficients of this lane's Q channels of the interval block at
// `off`, loaded once per run of neighbours that share the interval.
template <int Q>
__device__ __forceinline__ void fwd_load_cf(const FwdParams<float> &P, const float *__restrict__ tab, const int lane,
                                            const int off, float (&cf)[Q > 0 ? Q : 1][6]) {
  const float2 *q0 = reinterpret_cast<const float2 *>(tab + off) + lane;
  const float2 *q1 = q0 + P.M1, *q2 = q1 + P.M1;
#pragma unroll
  for (int k = 0; k < Q; ++k) {
    const float2 x = __ldg(q0 + 32 * k), y = __ldg(q1 + 32 * k), z = __ldg(q2 + 32 * k);
    cf[k][0] = x.x;
    cf[k][1] = x.y;
    cf[k][2] = y.x;
    cf[k][3] = y.y;
    cf[k][4] = z.x;
    cf[k][5] = z.y;
  }
}

// f32: one neighbour folded into the lane's Q channel rounds with the
// interval's coefficients already in registers.
template <int Q>
__device__ __forceinline__ void fwd_neighbour_cached(const float t, const float4 r, float (&acc)[Q > 0 ? Q : 1][4],
                                                     const float (&cf)[Q > 0 ? Q : 1][6]) {
#pragma unroll
  for (int k = 0; k < Q; ++k) {
    const float g = horner5(cf[k], t);
    acc[k][0] = fmaf(r.x, g, acc[k][0]);
    acc[k][1] = fmaf(r.y, g, acc[k][1]);
    acc[k][2] = fmaf(r.z, g, acc[k][2]);
    acc[k][3] = fmaf(r.w, g, acc[k][3]);
  }
}

// D_i = S_i (S_i^<)^T from T_i still in registers (Sec. II, the descriptor):
// D[m][n] = sum_k T[k][m] T[k][n], n < M2 <= 32.  T[k][n] for n < M2 is held
// by round 0, lane n (or, when M1 < 32, by remainder lane n) and reaches the
// other lanes by shuffles.  Main-round rows m = 32 r + lane are computed by
// their owners; the RR remainder rows are spread as (row, n) pairs over all
// 32 lanes so that no FMA instruction runs with a handful of lanes.
template <typename real, int Q>
__device__ __forceinline__ void descriptor_epilogue(const FwdParams<real> &P, const real (&acc)[Q > 0 ? Q : 1][4],
                                                   real rq0, real rq1, real rq2, real rq3, const int lane,
                                                   const int64_t i) {
  const int M1 = P.M1, M2 = P.M2;
  io_t<real> *__restrict__ Di = P.D + i * (int64_t)M1 * M2;
  for (int n = 0; n < M2; ++n) {  // uniform
    real t0, t1, t2, t3;
    if (Q > 0) {
      t0 = shfl(acc[0][0], n);
      t1 = shfl(acc[0][1], n);
      t2 = shfl(acc[0][2], n);
      t3 = shfl(acc[0][3], n);
    } else {
      t0 = shfl(rq0, n);
      t1 = shfl(rq1, n);
      t2 = shfl(rq2, n);
      t3 = shfl(rq3, n);
    }
#pragma unroll
    for (int r = 0; r < Q; ++r) {
      real d = acc[r][0] * t0;
      d = fma(acc[r][1], t1, d);
      d = fma(acc[r][2], t2, d);
      d = fma(acc[r][3], t3, d);
      Di[(size_t)(r * 32 + lane) * M2 + n] = to_io(d);
    }
  }
  const int npairs = P.RR * M2;
  for (int p0 = 0; p0 < npairs; p0 += 32) {  // uniform
    const int p = p0 + lane;
    const bool ok = p < npairs;
    const int j = ok ? p / M2 : 0, n = ok ? p - j * M2 : 0;
    const real a0 = shfl(rq0, j), a1 = shfl(rq1, j);
    const real a2 = shfl(rq2, j), a3 = shfl(rq3, j);
    real b0, b1, b2, b3;
    if (Q > 0) {
      b0 = shfl(acc[0][0], n);
      b1 = shfl(acc[0][1], n);
      b2 = shfl(acc[0][2], n);
      b3 = shfl(acc[0][3], n);
    } else {
      b0 = shfl(rq0, n);
      b1 = shfl(rq1, n);
      b2 = shfl(rq2, n);
      b3 = shfl(rq3, n);
    }
    real d = a0 * b0;
    d = fma(a1, b1, d);
    d = fma(a2, b2, d);
    d = fma(a3, b3, d);
    if (ok) Di[(size_t)(Q * 32 + j) * M2 + n] = to_io(d);
  }
}

// One atom: T_i into P.T (the whole warp takes part).  kMoments: runs of
// neighbours sharing an interval are contracted through their moments
//   W[k][q] = sum_{j in run} R~_j[k] t_j^q,   T[k][m] += sum_q C_{l,m,q} W[k][q]
// (C_{l,m,q} the t^q coefficient of channel m on interval l): the same sum as
// the per-neighbour evaluation, associated per interval.  A run that reaches
// the end of a 32-row batch keeps its partial W for the next batch, so that a
// run costs one T update however the batches cut it.
template <typename real, int Q, bool kMoments>
__device__ __forceinline__ void fwd_atom(const FwdParams<real> &P, Stage<real> &st, MomentStage<real> &ms,
                                         const int lane, const int64_t i) {
  constexpr bool kCache = sizeof(real) == 4;  // f32: coefficients reused along runs of equal intervals

  // valid rows per type segment (clamped into [0, sel]), kept in shared memory, and their total
  {
    int sl = 0;  // sel[lane] without indexing the parameter array dynamically
#pragma unroll
    for (int q = 0; q < DP_MAX_TYPES; ++q)
      if (lane == q) sl = P.sel[q];
    int x = 0;
    if (lane < P.ntypes) x = clampi(P.nvalid ? __ldg(P.nvalid + i * P.ntypes + lane) : sl, 0, sl);
    if (lane < DP_MAX_TYPES) st.nvb[lane] = x;
  }
  __syncwarp();
  int nv = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q) nv += st.nvb[q];
  const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
  const real *__restrict__ tab = P.table + (size_t)alpha * P.ntypes * P.pair_stride;
  const io_t<real> *__restrict__ srow = P.s + i * P.nnei;
  const io_t<real> *__restrict__ Rrow = P.Rt + i * P.nnei * 4;

  // packed-round role of this lane: neighbour slot and remainder channel
  const int rslot = P.RR > 0 ? lane / P.RR : 0;
  const int rch = P.RR > 0 ? lane - rslot * P.RR : 0;
  const bool ractive = P.RR > 0 && rslot < P.PK;

  real acc[Q > 0 ? Q : 1][4];
#pragma unroll
  for (int r = 0; r < (Q > 0 ? Q : 1); ++r) acc[r][0] = acc[r][1] = acc[r][2] = acc[r][3] = real(0);
  real racc0 = real(0), racc1 = real(0), racc2 = real(0), racc3 = real(0);
  real rcf[6];
  int rcur = -1;
  real cf[Q > 0 ? Q : 1][6];  // f32: coefficients of the interval in use
  // T += C_l W for the run in interval block `off`, W[6k + q] held by lanes 0..23 (uniform call)
  // remainder channels 32 Q + rch of the pending runs: lane (rslot, rch) takes run rslot (uniform call)
  int npend = 0;
  auto flush_remainder = [&]() {
    __syncwarp();
    if (ractive && rslot < npend) {
      real c6[6];
      ld6(tab + ms.poff[rslot], P.M1, Q * 32 + rch, c6);
      const real *w = ms.w[rslot];
      real v0 = racc0, v1 = racc1, v2 = racc2, v3 = racc3;
#pragma unroll
      for (int q = 0; q < 6; ++q) {
        v0 = fma(c6[5 - q], w[q], v0);
        v1 = fma(c6[5 - q], w[6 + q], v1);
        v2 = fma(c6[5 - q], w[12 + q], v2);
        v3 = fma(c6[5 - q], w[18 + q], v3);
      }
      racc0 = v0;
      racc1 = v1;
      racc2 = v2;
      racc3 = v3;
    }
    __syncwarp();
    npend = 0;
  };
  const int pend_cap = P.PK < kPendRuns ? P.PK : kPendRuns;
  auto apply_moments = [&](int off, real wv) {
    if (lane < 24) ms.w[npend][lane] = wv;
    if (lane == 0) ms.poff[npend] = off;
    __syncwarp();
    real W[4][6];
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
      for (int q = 0; q < 6; ++q) W[k][q] = ms.w[npend][6 * k + q];
#pragma unroll
    for (int r = 0; r < (Q > 0 ? Q : 1); ++r) {
      real c6[6];  // (a, b, c, d, e, f) = coefficients of t^5 .. t^0
      ld6(tab + off, P.M1, r * 32 + lane, c6);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        real v = acc[r][k];
#pragma unroll
        for (int q = 0; q < 6; ++q) v = fma(c6[5 - q], W[k][q], v);
        acc[r][k] = v;
      }
    }
    __syncwarp();
    if (P.RR > 0 && ++npend == pend_cap) flush_remainder();
  };
  int carry_off = -1;  // run left open at the end of the previous batch (uniform)
  real wcarry = real(0);  // its partial W on lanes 0..23
  for (int base = 0; base < nv; base += 32) {
    // stage: lane l prepares valid neighbour base + l
    const int v = base + lane;
    if (v < nv) {
      int b = 0, cum = 0, lim = st.nvb[0], off = 0;
#pragma unroll
      for (int q = 1; q < DP_MAX_TYPES; ++q)
        if (q < P.ntypes && v >= lim) {
          b = q;
          cum = lim;
          lim += st.nvb[q];
          off += P.sel[q - 1];
        }
      const int row = off + (v - cum);
      const Vec4<real> rr = ld4r<real>(Rrow + (size_t)row * 4);
      real t;
      bool clamped;
      const int l = locate(P.geom, __ldg(srow + row), t, clamped);
      st.r[lane][0] = rr.x;
      st.r[lane][1] = rr.y;
      st.r[lane][2] = rr.z;
      st.r[lane][3] = rr.w;
      st.t[lane] = t;
      st.off[lane] = (b * P.geom.nint + l) * P.M1 * 6;
      if constexpr (kMoments) {
        const real t2 = t * t, t3 = t2 * t;
        ms.tp[lane][0] = real(1);
        ms.tp[lane][1] = t;
        ms.tp[lane][2] = t2;
        ms.tp[lane][3] = t3;
        ms.tp[lane][4] = t2 * t2;
        ms.tp[lane][5] = t3 * t2;
      }
    }
    __syncwarp();
    const int cnt = min(32, nv - base);
    int nshort = cnt;  // rows whose remainder channels go through the packed per-neighbour round
    if (Q > 0 && kMoments) {
      nshort = 0;
      // W of a contracted run waiting for its T update (uniform): first the run left open by the
      // last batch if this batch does not continue it, then each contracted run of this batch.
      // The update has this one call site, so its (large) code is inlined once.
      int apply_off = -1;
      real apply_w = wcarry;
      if (carry_off >= 0 && st.off[0] != carry_off) {  // the open run ended with the last batch
        apply_off = carry_off;
        carry_off = -1;
      }
      int next_carry = -1;
      // run starts of the batch: rows whose interval block differs from the previous row's
      const int myoff = lane < cnt ? st.off[lane] : -1;
      const int prevoff = __shfl_up_sync(0xffffffffu, myoff, 1);
      unsigned starts = __ballot_sync(0xffffffffu, lane < cnt && (lane == 0 || myoff != prevoff));
      while (starts || apply_off >= 0) {  // uniform, run by run
        if (apply_off >= 0) {
          apply_moments(apply_off, apply_w);
          apply_off = -1;
          continue;
        }
        const int u = __ffs(starts) - 1;
        starts &= starts - 1;
        const int e = starts ? __ffs(starts) - 1 : cnt;
        const int off = __shfl_sync(0xffffffffu, myoff, u);
        const bool cont = u == 0 && off == carry_off;
        if (cont || e - u >= min_moment_run<real>()) {
          real wv = cont ? wcarry : real(0);
          if (lane < 24) {
            const int k = lane / 6, q = lane - 6 * (lane / 6);
            for (int j = u; j < e; ++j) wv = fma(st.r[j][k], ms.tp[j][q], wv);
          }
          if (e == cnt && base + 32 < nv) {  // may go on in the next batch: keep W open
            wcarry = wv;
            next_carry = off;
          } else {
            apply_off = off;
            apply_w = wv;
          }
        } else {
          for (int j = u; j < e; ++j) fwd_neighbour<real, Q>(P, tab, lane, off, st.t[j], st.r[j], acc);
          if (lane >= u && lane < e) ms.srow[nshort + lane - u] = lane;  // their remainder channels: packed round
          nshort += e - u;
        }
      }
      carry_off = next_carry;
    } else if (Q > 0) {
      if constexpr (kCache) {
        // f32: walk the batch run by run.  Neighbours are sorted by distance
        // inside a type segment, so consecutive ones often share an interval:
        // its coefficients are loaded once at the start of the run (a real
        // branch, not loads predicated on every neighbour) and reused.
        int u = 0;
        while (u < cnt) {  // uniform
          const int off = st.off[u];
          fwd_load_cf<Q>(P, tab, lane, off, cf);
          do {
            fwd_neighbour_cached<Q>(st.t[u], *reinterpret_cast<const float4 *>(st.r[u]), acc, cf);
            ++u;
          } while (u < cnt && st.off[u] == off);
        }
      } else {
        for (int u = 0; u < cnt; ++u)  // uniform: every lane on neighbour u
          fwd_neighbour<real, Q>(P, tab, lane, st.off[u], st.t[u], st.r[u], acc);
      }
    }
    if (P.RR > 0) {
      __syncwarp();
      for (int u0 = 0; u0 < nshort; u0 += P.PK) {  // packed round: PK neighbours x RR channels
        const int x = u0 + rslot;
        if (ractive && x < nshort) {
          const int u = (Q > 0 && kMoments) ? ms.srow[x] : x;
          const real t = st.t[u];
          const int off = st.off[u];
          if (!kCache || off != rcur) {
            rcur = off;
            ld6(tab + off, P.M1, Q * 32 + rch, rcf);
          }
          const real g = horner5(rcf, t);
          racc0 = fma(st.r[u][0], g, racc0);
          racc1 = fma(st.r[u][1], g, racc1);
          racc2 = fma(st.r[u][2], g, racc2);
          racc3 = fma(st.r[u][3], g, racc3);
        }
      }
    }
    __syncwarp();
  }

  if (Q > 0 && kMoments && npend > 0) flush_remainder();

  io_t<real> *__restrict__ Ti = P.T + i * 4 * P.M1;
#pragma unroll
  for (int r = 0; r < Q; ++r) {
#pragma unroll
    for (int k = 0; k < 4; ++k) acc[r][k] *= P.inv_nnei;  // acc now holds T_i
    const int m = r * 32 + lane;
    Ti[m] = to_io(acc[r][0]);
    Ti[P.M1 + m] = to_io(acc[r][1]);
    Ti[2 * P.M1 + m] = to_io(acc[r][2]);
    Ti[3 * P.M1 + m] = to_io(acc[r][3]);
  }
  if (P.RR > 0) {
    // lanes rch, rch + RR, ..., rch + (PK-1) RR hold partial sums of channel 32 Q + rch
    for (int k = 1; k < P.PK; ++k) {
      const int src = lane + k * P.RR;
      const real x0 = shfl(racc0, src & 31), x1 = shfl(racc1, src & 31);
      const real x2 = shfl(racc2, src & 31), x3 = shfl(racc3, src & 31);
      if (lane < P.RR) {
        racc0 += x0;
        racc1 += x1;
        racc2 += x2;
        racc3 += x3;
      }
    }
    racc0 *= P.inv_nnei;
    racc1 *= P.inv_nnei;
    racc2 *= P.inv_nnei;
    racc3 *= P.inv_nnei;
    if (lane < P.RR) {
      const int m = Q * 32 + lane;
      Ti[m] = to_io(racc0);
      Ti[P.M1 + m] = to_io(racc1);
      Ti[2 * P.M1 + m] = to_io(racc2);
      Ti[3 * P.M1 + m] = to_io(racc3);
    }
  }
  if constexpr (!kMoments)  // the fused descriptor is offered with the per-row forward only
    if (P.D) descriptor_epilogue<real, Q>(P, acc, racc0, racc1, racc2, racc3, lane, i);
}

template <typename real, int Q, bool kMoments>
__global__ void __launch_bounds__(kFwdWarps * 32) fwd_kernel(const FwdParams<real> P) {
  __shared__ Stage<real> stage[kFwdWarps];
  __shared__ MomentStage<real> mstage[kMoments ? kFwdWarps : 1];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t i = (int64_t)blockIdx.x * kFwdWarps + w;
  if (i < P.nloc) fwd_atom<real, Q, kMoments>(P, stage[w], mstage[kMoments ? w : 0], lane, i);  // warp-uniform
}

template <typename real>
using FwdKernel = void (*)(const FwdParams<real>);

template <typename real, bool kMoments, int... Qs>
FwdKernel<real> pick_fwd(int Q, std::integer_sequence<int, Qs...>) {
  FwdKernel<real> k = nullptr;
  ((Q == Qs ? (k = &fwd_kernel<real, Qs, kMoments>, 0) : 0), ...);
  return k;
}

template <typename real>
int fwd(const real *table, const dp_table_info *info, const io_t<real> *s, const io_t<real> *Rt,
        const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1,
        io_t<real> *T, void *stream, int M2 = 0, io_t<real> *D = nullptr, bool want_D = false,
        bool moments = false) {
  clear_error();
  TableGeom g;
  Segments seg;
  int rc = check_fusion_args(table, info, s, Rt, nloc, nnei, ntypes, sel, M1, T, want_D ? (const void *)D : T, &g,
                             &seg);
  if (rc) return rc;
  if (want_D) {
    if (M2 < 1 || M2 > M1) return set_error(DP_ERR_SHAPE, "need 1 <= M2 <= M1 (M1 %d, M2 %d)", M1, M2);
    if (M2 > 32) return set_error(DP_ERR_UNSUPPORTED, "fused descriptor needs M2 <= 32 (M2 = %d)", M2);
  }
  if (nloc == 0) return DP_OK;
  FwdParams<real> P;
  P.table = table;
  P.s = s;
  P.Rt = Rt;
  P.nvalid = nvalid;
  P.atype = atype;
  P.T = T;
  P.D = want_D ? D : nullptr;
  P.M2 = want_D ? M2 : 0;
  P.geom = GeomOf<real>::make(g);
  P.nloc = nloc;
  P.nnei = nnei;
  P.ntypes = ntypes;
  P.M1 = M1;
  P.pair_stride = g.nint * M1 * 6;
  const int Q = M1 / 32;
  P.RR = M1 - 32 * Q;
  P.PK = P.RR > 0 ? 32 / P.RR : 1;
  for (int b = 0; b < DP_MAX_TYPES; ++b) P.sel[b] = seg.sel[b];
  P.inv_nnei = host_cvt<real>(1.0 / (double)nnei);
  FwdKernel<real> k = nullptr;
  if (moments)
    k = pick_fwd<real, true>(Q, std::make_integer_sequence<int, DP_MAX_M1 / 32 + 1>{});
  else if constexpr (!std::is_same<real, df64>::value)  // df64 runs the moment form only
    k = pick_fwd<real, false>(Q, std::make_integer_sequence<int, DP_MAX_M1 / 32 + 1>{});
  if (!k) return set_error(DP_ERR_UNSUPPORTED, "no forward kernel for M1 = %d", M1);
  const int64_t blocks = (nloc + kFwdWarps - 1) / kFwdWarps;
  if (blocks > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
  k<<<(unsigned)blocks, kFwdWarps * 32, 0, (cudaStream_t)stream>>>(P);
  return launch_status("dp_tabulate_fusion_fwd");
}

}  // namespace

}  // namespace dpc

extern "C" {

int dp_tabulate_fusion_fwd_f64(const double *table, const dp_table_info *info, const double *s, const double *Rt,
                               const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                               const int32_t *sel, int M1, double *T, void *stream) {
  return dpc::fwd<double>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, stream);
}

int dp_tabulate_fusion_fwd_f32(const float *table, const dp_table_info *info, const float *s, const float *Rt,
                               const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                               const int32_t *sel, int M1, float *T, void *stream) {
  return dpc::fwd<float>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, stream);
}

int dp_tabulate_fusion_fwd_moments_f64(const double *table, const dp_table_info *info, const double *s,
                                       const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                       int nnei, int ntypes, const int32_t *sel, int M1, double *T, void *stream) {
  return dpc::fwd<double>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, stream, 0, nullptr, false,
                          true);
}

int dp_tabulate_fusion_fwd_moments_f32(const float *table, const dp_table_info *info, const float *s,
                                       const float *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                       int nnei, int ntypes, const int32_t *sel, int M1, float *T, void *stream) {
  return dpc::fwd<float>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, stream, 0, nullptr, false,
                         true);
}

int dp_tabulate_fusion_fwd_moments_df64(const float *table, const dp_table_info *info, const double *s,
                                        const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                        int nnei, int ntypes, const int32_t *sel, int M1, double *T, void *stream) {
  return dpc::fwd<dpc::df64>(reinterpret_cast<const dpc::df64 *>(table), info, s, Rt, nvalid, atype, nloc, nnei,
                             ntypes, sel, M1, T, stream, 0, nullptr, false, true);
}

int dp_tabulate_fusion_fwd_descriptor_f64(const double *table, const dp_table_info *info, const double *s,
                                          const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                          int nnei, int ntypes, const int32_t *sel, int M1, int M2, double *T,
                                          double *D, void *stream) {
  return dpc::fwd<double>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, stream, M2, D, true);
}

int dp_tabulate_fusion_fwd_descriptor_f32(const float *table, const dp_table_info *info, const float *s,
                                          const float *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                          int nnei, int ntypes, const int32_t *sel, int M1, int M2, float *T,
                                          float *D, void *stream) {
  return dpc::fwd<float>(table, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, stream, M2, D, true);
}

}  // extern "C"
