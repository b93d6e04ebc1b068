// Persistent exact-f64 GEMM for the tensor-core tabulation (tabulate_tc.cu): the per-interval
// contraction of every 12-atom tile in the forward (T = W C' over the used K slices), on the 9 x 6-bit
// digit-split operands of tc_gemm.cuh; also the backward (dW = dT C'^T over the used 128-row output
// tiles) where M1 > 144 (else tab_gemm_b8.cuh's 7 x 8-bit kernel runs it).
//
// One CTA per SM walks its units: forward, the pieces the schedule gave it, in order -- (centre type,
// atom tile, 128-row tile of A, a run of at most 112 of the tile's used slices), every centre type in
// one launch; backward, a list of the (atom tile, 128-row output tile) pairs with work, round-robin
// over the grid.  The TMEM accumulators (nine diagonals x 48 columns), the mbarriers and the stage ring
// are set up once per CTA, and the roles run ahead of each other: warp 0 moves each slice's A block
// (and in the backward its B block) into a ring of four stages (bulk copies counted on the stage's
// "full" barrier); in the forward a split warp per stage writes the B block from the moments, as digit
// planes, and arrives on the same barrier; lane 0 of warp 1 issues the slice's 13 MMAs and frees the
// stage ("empty") when they complete; eight epilogue warps (two per TMEM lane quadrant, 24 columns
// each) read the unit's accumulators once its last MMA has completed ("acc_full"), recombine each
// output's diagonals exactly as an integer and round it once to f64 (diag_to_f64) -- or, for a piece
// of a cut item, store the integer for fwd_finish_kernel to sum -- write the outputs, then release
// the accumulators ("tmem_free") for the next unit's MMAs.  The copies of the next unit overlap the
// epilogue of this one.  The two directions are separate instantiations of the kernel.
// Every wait is bounded; a wait that gives up stops the CTA's copies and MMAs, its remaining
// outputs are NaN and one timeout is counted (dp_tc_wait_timeouts).
#pragma once

#include "tc_gemm.cuh"

namespace dpc {
namespace {
namespace tg {
using namespace tc;

constexpr int kEpiWarps = 8;    // two per TMEM lane quadrant
constexpr long long kPartNaN = 1ll << 62;  // high word of a piece's output whose accumulators were not read
constexpr int kSplitWarps = 4;  // forward: the B digit planes of each slice, made in shared memory
constexpr int kThreadsP = 32 * (2 + kEpiWarps + kSplitWarps);  // producer, MMA issuer, epilogue, split warps
constexpr int kEpiCols = kTN / 2;              // columns per epilogue warp
constexpr int kMaxUnitSlices = kMaxShareSlices;
constexpr int kTileAtomsP = kTN / 4;  // atoms per tile (four columns each)

struct Params {
  bool fwd;
  // A: blocks [Mp / 128][ka] of kS x kPlaneA bytes; E: [Mp] row exponents
  const unsigned char *aplanes;
  const int *Eexp;
  int ka;   // K slices per row of blocks (forward: every K slice of the table; backward: M1 / 16)
  int nmt;  // 128-row tiles of A
  // B: blocks [ntiles][ka] of kS x kPlaneB bytes, or (W != NULL) made by the split warps from the
  // moments W[natoms][cap][24] and the run map [natoms][nkeys]; F: [Np] column exponents
  const unsigned char *bplanes;
  const double *W;
  const int *map;
  const int *Fexp;
  int64_t ntiles, Np, Mp;
  // forward: the tile's used slices, in order ([ntiles][ka] and [ntiles]), in shares of 28
  const short *slist;
  const int *scount;
  int zmax;
  longlong2 *part;  // [slot][48][Mp]: exact integers (lo, hi) of the pieces of cut items (see diag_s128)
  double *tout;  // T, written by tiles with one share: [(atom0 + a) 4 + k][ldt]
  int ldt;
  // backward: output tile (tile, mt) wanted when one of K slices 8 mt .. 8 mt + 7 is flagged
  const unsigned char *sflags;  // [ntiles][nsf]
  int nsf;
  double *scat;  // [natoms][cap][24]: the wanted outputs, per run slot, finished to f64
  const short *keys;
  const int *nslots;
  int cap, nkeys, kq;
  // forward, every centre type in one launch: the pieces of work (int4: tile; type | mt << 4 | slices << 8;
  // first slice in the tile's list; part slot, or -1 for a tile whose T the piece writes itself), CTA b
  // taking pieces cta_start[b] .. cta_start[b + 1] - 1 in order; per type, the A planes lie astride
  // bytes apart, the row exponents estride apart, the slice lists and counts ntiles ka and ntiles apart
  const int4 *pieces;
  const int *cta_start;
  size_t astride;
  int estride;
  // both
  const int32_t *atype;
  int64_t natoms, atom0;
  int alpha, ntypes;  // backward: the launch's centre type
  const int *units;   // backward: the launch's units, packed (unit_code), in any order
  const int *nunits;  // their count (device)
};

// A unit packed into an int: tile (< 2^16), 128-row tile of A (< 2^8), share (< 2^8).
__host__ __device__ constexpr int unit_code(int tile, int mt, int z) { return tile | (mt << 16) | (z << 24); }

struct Unit {
  int64_t tile;
  int alpha, mt, s0, nsl, slot;  // centre type, 128-row tile of A, first slice and slice count, part slot
};

// Unit i of the CTA's walk (every role walks the same units).
template <bool kFwd>
__device__ __forceinline__ Unit unit_of(const Params &P, int i) {
  Unit U;
  if (kFwd) {
    const int4 c = P.pieces[i];
    U.tile = c.x;
    U.alpha = c.y & 15;
    U.mt = (c.y >> 4) & 15;
    U.nsl = c.y >> 8;
    U.s0 = c.z;
    U.slot = c.w;
  } else {
    const int c = P.units[i];
    U.tile = c & 0xffff;
    U.alpha = P.alpha;
    U.mt = (c >> 16) & 0xff;
    U.nsl = P.ka;
    U.s0 = 0;
    U.slot = -1;
  }
  return U;
}

// The CTA's units: forward its pieces in order, backward the launch's list round-robin.
struct Walk {
  int begin, end, step;
};
template <bool kFwd>
__device__ __forceinline__ Walk walk_of(const Params &P) {
  if (kFwd) return Walk{P.cta_start[blockIdx.x], P.cta_start[blockIdx.x + 1], 1};
  return Walk{(int)blockIdx.x, *P.nunits, (int)gridDim.x};
}

// A wait on an mbarrier phase, bounded in time (2 s on the global timer), that also gives up once another
// role has.  The waiting thread is suspended between polls (try_wait's time hint), so that a waiting
// thread takes no issue slots or shared-memory bandwidth from the copies and the MMAs.
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, volatile int *abortf) {
  const uint64_t t0 = global_ns();
  for (;;) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(done)
        : "r"(bar), "r"(parity), "r"(20000u)
        : "memory");
    if (done) return true;
    if (*abortf) return false;
    if (global_ns() - t0 > 2000000000ull) {
      *abortf = 1;
      return false;
    }
  }
}

constexpr size_t kBarOff = (size_t)kStages * kStageBytes;  // full[4], empty[4], acc_full, tmem_free
constexpr size_t kMiscOff = kBarOff + (2 * kStages + 2) * 8;  // tmem address, abort flag
constexpr size_t kListOff = kMiscOff + 16;                     // producer's slice list
constexpr size_t kStabOff = kListOff + kMaxUnitSlices * 4;     // epilogue: slot table, slot counts, flags
constexpr size_t kSmemP = kStabOff + (kScatKeys * kScatAtoms + 2 * kScatAtoms + 4 + kTN) * 4;
static_assert(kSmemP <= 227 * 1024, "shared memory per block");

// kFwd: the forward (B made from the moments by the split warps, pieces in order); else the backward
// (B copied from its digit planes, units round-robin).  Two instantiations, each carrying only its own
// code (measured: one kernel with both directions stalled on instruction fetch).
template <bool kFwd>
__global__ void __launch_bounds__(kThreadsP, 1) tgemm_kernel(const Params P) {
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + kBarOff);
  uint64_t *empty = full + kStages;
  uint64_t *acc_full = empty + kStages;
  uint64_t *tmem_free = acc_full + 1;
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(smem + kMiscOff);
  volatile int *abortf = reinterpret_cast<volatile int *>(smem + kMiscOff + 4);
  int *plist = reinterpret_cast<int *>(smem + kListOff);
  int *stab = reinterpret_cast<int *>(smem + kStabOff);  // (key of the tile, atom) -> slot
  int *nsa = stab + kScatKeys * kScatAtoms;                // per atom: slot count (backward) or wanted (forward)
  int *uflag = nsa + 2 * kScatAtoms;  // [0]: the unit writes T directly; [1]: its accumulators are ready
  int *fexp_s = uflag + 4;             // the unit's 48 column exponents
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const Walk wk = walk_of<kFwd>(P);

  constexpr bool fused = kFwd;  // B made in shared memory by the split warps
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(full + s)), "r"(fused ? 2 : 1));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(empty + s)));
    }
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(acc_full)));
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(tmem_free)), "r"(kEpiWarps));
    asm volatile("fence.mbarrier_init.release.cluster;");
    *abortf = 0;
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

  if (warp == 0) {
    // ---- producer: each slice's A and B blocks into the next stage of the ring
    int g = 0;  // slices loaded so far by this CTA
    for (int u = wk.begin; u < wk.end; u += wk.step) {
      if (__shfl_sync(0xffffffffu, (int)*abortf, 0)) break;  // uniform over the warp
      const Unit U = unit_of<kFwd>(P, u);
      if (kFwd)
        for (int j = lane; j < U.nsl; j += 32)
          plist[j] = P.slist[((size_t)U.alpha * P.ntiles + U.tile) * P.ka + U.s0 + j];
      __syncwarp();
      if (lane == 0) {
        for (int j = 0; j < U.nsl; ++j, ++g) {
          const int sl = kFwd ? plist[j] : j;
          const int st = g % kStages;
          if (g >= kStages && !wait_or_abort(smem_u32(empty + st), (uint32_t)((g / kStages - 1) & 1), abortf)) break;
          const unsigned char *asrc = P.aplanes + U.alpha * P.astride + ((size_t)U.mt * P.ka + sl) * (kS * kPlaneA);
          const unsigned char *bsrc = P.bplanes + ((size_t)U.tile * P.ka + sl) * (kS * kPlaneB);
          const uint32_t bar = smem_u32(full + st), dst = sbase + st * kStageBytes;
          const uint32_t bytes = fused ? kS * kPlaneA : kStageBytes;
          asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
              "l"(asrc), "r"((uint32_t)(kS * kPlaneA)), "r"(bar)
              : "memory");
          if (!fused)
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    dst + kS * kPlaneA),
                "l"(bsrc), "r"((uint32_t)(kS * kPlaneB)), "r"(bar)
                : "memory");
        }
      }
      g = __shfl_sync(0xffffffffu, g, 0);
      __syncwarp();  // the list is reused by the next unit
    }
  } else if (warp == 1) {
    // ---- MMA issuer: per slice the 45 digit products as 13 MMAs (see gemm_kernel), per unit a commit
    // on acc_full once they have all completed
    if (lane == 0) {
      int g = 0, li = 0;
      bool ok = true;
      for (int u = wk.begin; u < wk.end && ok; u += wk.step) {
        const Unit U = unit_of<kFwd>(P, u);
        if (li > 0 && !(ok = wait_or_abort(smem_u32(tmem_free), (uint32_t)((li - 1) & 1), abortf))) break;
        asm volatile("tcgen05.fence::after_thread_sync;");
        for (int j = 0; j < U.nsl; ++j, ++g) {
          const int st = g % kStages;
          if (!(ok = wait_or_abort(smem_u32(full + st), (uint32_t)((g / kStages) & 1), abortf))) break;
          asm volatile("tcgen05.fence::after_thread_sync;");
          const uint64_t a0 = smem_desc(sbase + st * kStageBytes), b0 = smem_desc(sbase + st * kStageBytes + kS * kPlaneA);
#pragma unroll
          for (int s = 0; s < kS; ++s) {
            const uint64_t ad = a0 + (uint64_t)((s * kPlaneA) >> 4);
#pragma unroll
            for (int t0 = 0; t0 < kS - s; t0 += kMaxPlanesPerMma) {
              const int np = min(kMaxPlanesPerMma, kS - s - t0);
              const uint64_t bd = b0 + (uint64_t)((t0 * kPlaneB) >> 4);
              const uint32_t idesc = kIdescNoN | ((uint32_t)((np * kTN) >> 3) << 17);
              const uint32_t acc = (j > 0 || s > 0) ? 1u : 0u;  // a unit's first digit product writes every diagonal
              asm volatile(
                  "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                  " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem + (uint32_t)((s + t0) * kTN)),
                  "l"(ad), "l"(bd), "r"(idesc), "r"(acc));
            }
          }
          asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
              smem_u32(empty + st)));
        }
        // completes when every MMA issued so far has (also after a wait that gave up)
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(acc_full)));
        ++li;
      }
    }
    __syncwarp();
  } else if (warp >= 2 + kEpiWarps) {
    // ---- split warps (forward): each slice's B block -- B[6 key + q][4 a + k] = W_a[k][(key, q)], the
    // moments of the atom's run slot of that interval -- as balanced digit planes in the stage, in the
    // tcgen05 K-major core-matrix layout.  Warp w owns stage w (the slices g with g % 4 == w), so four
    // slices are made at once.  Lane (k = lane / 8, kp = lane % 8) makes the K entries 2 kp, 2 kp + 1 of
    // column 4 i + k for the tile's atoms i = 0 .. 11 (one key per lane and slice, 6 being even): the
    // column exponents and the unit's slice list are read once per unit, the run slots of the warp's
    // next slice are loaded while this slice's moments are, and the stage is waited for only before
    // the stores; then a fence makes the writes visible to the tensor core and the warp arrives on the
    // stage's "full" barrier.  (Measured: with a global load chain per slice the tensor core waited
    // ~0.6 us per slice for its B block.)
    static_assert(kSplitWarps == kStages, "a split warp per stage");
    if (fused) {
      const int w = warp - (2 + kEpiWarps);
      constexpr int kPairs = kTileAtomsP;  // per lane and slice: one pair of K entries per atom
      static_assert(kTN * kTK / 2 == 32 * kPairs, "a pair per lane and atom");
      const int k = lane >> 3, kp = lane & 7;
      int g0 = 0;  // slices of this CTA before the unit
      for (int u = wk.begin; u < wk.end; u += wk.step) {
        if (__shfl_sync(0xffffffffu, (int)*abortf, 0)) break;  // uniform over the warp
        const Unit U = unit_of<kFwd>(P, u);
        const int64_t a_base = (int64_t)U.tile * kTileAtomsP;
        const short *ulist = P.slist + ((size_t)U.alpha * P.ntiles + U.tile) * P.ka + U.s0;
        int E[kPairs];
        bool av[kPairs];
#pragma unroll
        for (int i = 0; i < kPairs; ++i) {
          E[i] = P.Fexp[U.tile * kTN + 4 * i + k];
          av[i] = a_base + i < P.natoms;
        }

        auto load_slots = [&](int sl, int (&slot)[kPairs]) {
          const int key = (sl * kTK + 2 * kp) / 6;
#pragma unroll
          for (int i = 0; i < kPairs; ++i)
            slot[i] = (av[i] && key < P.nkeys) ? P.map[(a_base + i) * P.nkeys + key] : -1;
        };
        int j = ((w - g0) % kStages + kStages) % kStages;  // the warp's first slice of the unit
        // the warp's slices of the unit (at most 112 / 4 = 28): lane l holds entry j + 4 l of the list
        static_assert(kMaxUnitSlices / kStages <= 32, "a lane per slice of the warp");
        const int slr = j + kStages * lane < U.nsl ? ulist[j + kStages * lane] : 0;
        const int j_first = j;
        auto slice_at = [&](int jj) { return __shfl_sync(0xffffffffu, slr, ((jj - j_first) / kStages) & 31); };
        int sl = j < U.nsl ? __shfl_sync(0xffffffffu, slr, 0) : 0;
        int slot[kPairs], slotn[kPairs];
        if (j < U.nsl) load_slots(sl, slot);
        bool ok = true;
        for (; j < U.nsl; j += kStages) {
          const int g = g0 + j;
          const int jn = j + kStages;
          const int sln = jn < U.nsl ? slice_at(jn) : 0;
          if (jn < U.nsl) load_slots(sln, slotn);  // the next slice's slots, in flight with these moments
          const int kk = sl * kTK + 2 * kp, q0 = kk - 6 * (kk / 6);
          double2 xv[kPairs];
#pragma unroll
          for (int i = 0; i < kPairs; ++i)
            xv[i] = slot[i] >= 0
                        ? *reinterpret_cast<const double2 *>(P.W + ((size_t)(a_base + i) * P.cap + slot[i]) * 24 + 6 * k + q0)
                        : make_double2(0.0, 0.0);
          if (g >= kStages) {
            int wv = 1;
            if (lane == 0) wv = wait_or_abort(smem_u32(empty + w), (uint32_t)((g / kStages - 1) & 1), abortf);
            ok = __shfl_sync(0xffffffffu, wv, 0) != 0;
            if (!ok) break;
          }
          unsigned char *bstage = smem + w * kStageBytes + kS * kPlaneA;
#pragma unroll
          for (int i = 0; i < kPairs; ++i) {
            const int r = 4 * i + k;
            uint32_t h[kS];
            digit_pairs(biased_fixed(xv[i].x, E[i]), biased_fixed(xv[i].y, E[i]), h);
            unsigned char *dst = bstage + (r >> 3) * kSBO + (r & 7) * 16 + (kp >> 2) * kLBO + (kp & 3) * 4;
#pragma unroll
            for (int d = 0; d < kS; ++d) *reinterpret_cast<uint32_t *>(dst + d * kPlaneB) = h[d];
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          __syncwarp();
          if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(full + w)) : "memory");
          sl = sln;
#pragma unroll
          for (int i = 0; i < kPairs; ++i) slot[i] = slotn[i];
        }
        if (!ok) break;
        g0 += U.nsl;
      }
    }
  } else {
    // ---- epilogue: warps 2 .. 9, TMEM lane quadrant warp % 4, columns 24 ((warp - 2) / 4) .. + 23
    const int et = tid - 64;
    const int q = warp & 3, c_lo = ((warp - 2) / 4) * kEpiCols;
    const int rl = 32 * q + lane;
    const uint32_t trow = tmem + ((uint32_t)(32 * q) << 16);
    int li = 0;
    for (int u = wk.begin; u < wk.end; u += wk.step) {
      const Unit U = unit_of<kFwd>(P, u);
      const int64_t m0 = (int64_t)U.mt * kTM;
      const int n0 = (int)(U.tile * kTN);
      asm volatile("bar.sync 1, %0;" ::"r"(32 * kEpiWarps));  // the previous unit's tables are free
      if (et < kTN) fexp_s[et] = P.Fexp[n0 + et];
      if (kFwd) {
        if (et < kScatAtoms) {
          const int64_t a = (int64_t)(n0 / 4) + et;
          nsa[et] = a < P.natoms && (!P.atype || clampi(P.atype[P.atom0 + a], 0, P.ntypes - 1) == U.alpha);
        }
        if (et == 0) uflag[0] = P.tout && U.slot < 0;
      } else {
        for (int x = et; x < kScatKeys * kScatAtoms; x += 32 * kEpiWarps) stab[x] = -1;
        if (et < kScatAtoms) {
          const int64_t a = (int64_t)(n0 / 4) + et, i = P.atom0 + a;
          nsa[et] = a < P.natoms && (!P.atype || clampi(P.atype[i], 0, P.ntypes - 1) == P.alpha) ? P.nslots[i] : 0;
        }
        asm volatile("bar.sync 1, %0;" ::"r"(32 * kEpiWarps));
        const int key0 = (int)(m0 / P.kq);
        for (int al = et >> 5; al < kScatAtoms; al += kEpiWarps) {  // a warp per atom, its lanes over the slots
          const short *keys = P.keys + (P.atom0 + n0 / 4 + al) * P.cap;
          for (int slot = lane; slot < nsa[al]; slot += 32) {
            const int key = keys[slot];
            if (key >= key0 && key < key0 + kScatKeys) stab[(key - key0) * kScatAtoms + al] = slot;
          }
        }
      }
      if (et == 0) uflag[1] = !*abortf && wait_or_abort(smem_u32(acc_full), (uint32_t)(li & 1), abortf);
      asm volatile("bar.sync 1, %0;" ::"r"(32 * kEpiWarps));  // the tables are built and the MMAs done
      const bool ok = uflag[1] != 0;
      asm volatile("tcgen05.fence::after_thread_sync;");
      const bool direct = kFwd && uflag[0];
      const int Erow = (direct && m0 + rl < P.ldt) || (!kFwd && m0 + rl < P.Mp) ? P.Eexp[U.alpha * P.estride + m0 + rl] : 0;
      const int key = kFwd ? 0 : (int)((m0 + rl) / P.kq), qq = kFwd ? 0 : (int)(m0 + rl - (int64_t)key * P.kq);
      const int key_l = kFwd ? 0 : key - (int)(m0 / P.kq);
      const bool row_wanted = !kFwd && qq < 6 && key < P.nkeys;
      longlong2 *outp = kFwd && !direct ? P.part + (size_t)U.slot * kTN * P.Mp + m0 + rl : nullptr;
      // the warp's 24 columns of accumulators, four (one atom) at a time: each output's nine diagonals
      // recombined exactly as an integer and rounded once to f64 (diag_to_f64: integer operations, no
      // branch, the four outputs interleaved), or kept as four floats for a tile with several shares.
      // One copy of the loop body, so that it stays in the instruction cache (measured: two copies of
      // it, or two conversion variants, made the epilogue several times slower).
#pragma unroll 1
      for (int c0 = 0; c0 < kEpiCols; c0 += 4) {
        float v[kS][4];
        if (ok) {  // uniform over the CTA
#pragma unroll
          for (int d = 0; d < kS; ++d)
            asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
                         : "=f"(v[d][0]), "=f"(v[d][1]), "=f"(v[d][2]), "=f"(v[d][3])
                         : "r"(trow + (uint32_t)(d * kTN + c_lo + c0)));
          asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
          for (int d = 0; d < kS; ++d) asm volatile("" : "+f"(v[d][0]), "+f"(v[d][1]), "+f"(v[d][2]), "+f"(v[d][3]));
        }
        const int al = (c_lo + c0) >> 2;  // the group's atom; column c0 + k is its component k
        if (outp) {  // a piece of a cut item: its outputs' exact integers, summed by fwd_finish_kernel
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            long long hi;
            unsigned long long lo;
            diag_s128(v, k, hi, lo);
            outp[(size_t)(c_lo + c0 + k) * P.Mp] = ok ? make_longlong2((long long)lo, hi) : make_longlong2(0, kPartNaN);
          }
          continue;
        }
        // only the wanted outputs are stored; a warp skips a group none of its rows wants
        int64_t at = -1, ldk = 0;
        if (direct) {
          if (m0 + rl < P.ldt && nsa[al]) at = (P.atom0 + (int64_t)(n0 >> 2) + al) * 4 * P.ldt + m0 + rl, ldk = P.ldt;
        } else if (row_wanted) {
          const int slot = stab[key_l * kScatAtoms + al];
          if (slot >= 0) at = ((int64_t)((n0 >> 2) + al) * P.cap + slot) * 24 + qq, ldk = 6;
        }
        if (!__any_sync(0xffffffffu, at >= 0)) continue;
        double val[4];
        int F[4];
        bool rare = false;
#pragma unroll
        for (int k = 0; k < 4; ++k) F[k] = fexp_s[c_lo + c0 + k];
#pragma unroll
        for (int k = 0; k < 4; ++k) val[k] = diag_to_f64(v, k, Erow, F[k], rare);
        if (__any_sync(0xffffffffu, rare))  // warp-uniform, and never taken with these operands
#pragma unroll
          for (int k = 0; k < 4; ++k)
            val[k] = output_value_rare(v[0][k], v[1][k], v[2][k], v[3][k], v[4][k], v[5][k], v[6][k], v[7][k], v[8][k],
                                       Erow, F[k], false);
        if (at >= 0) {
          double *dst = (direct ? P.tout : P.scat) + at;
#pragma unroll
          for (int k = 0; k < 4; ++k) dst[k * ldk] = ok ? val[k] : __longlong_as_double(0x7ff8000000000000ll);
        }
      }
      asm volatile("tcgen05.fence::before_thread_sync;");
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(tmem_free)) : "memory");
      ++li;
    }
  }

  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  if (tid == 0 && *abortf) atomicAdd(&g_wait_timeouts, 1u);
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

// The kernels' shared-memory size, set once per device (bit d of set_on: done on device d).
int set_smem(const char *who) {
  static std::atomic<unsigned long long> set_on{0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(cudaGetLastError()));
  if (dev < 64 && (set_on.load(std::memory_order_acquire) >> dev & 1ull)) return DP_OK;
  for (const void *k : {(const void *)tgemm_kernel<true>, (const void *)tgemm_kernel<false>}) {
    const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemP);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
  }
  if (dev < 64) set_on.fetch_or(1ull << dev, std::memory_order_acq_rel);
  return DP_OK;
}

// One launch: grid CTAs (forward: the schedule's CTA count), or one per SM (backward, grid 0).
int launch(const Params &P, cudaStream_t st, const char *who, int grid = 0) {
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(cudaGetLastError()));
  if (P.fwd)
    tgemm_kernel<true><<<(unsigned)std::max(grid > 0 ? grid : nsm, 1), kThreadsP, kSmemP, st>>>(P);
  else
    tgemm_kernel<false><<<(unsigned)std::max(grid > 0 ? grid : nsm, 1), kThreadsP, kSmemP, st>>>(P);
  return launch_status(who);
}

}  // namespace tg
}  // namespace
}  // namespace dpc
