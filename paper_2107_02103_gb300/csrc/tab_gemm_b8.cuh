// Persistent exact-f64 GEMM for the tensor-core tabulation's backward where the channels fit one
// share of the 7 x 8-bit digit scheme (M1 <= 144): dW = dT C'^T over the used 128-row output tiles of
// every 8-atom tile, each output scattered to its atom's run slot (the rows kernel reads it there).
//
// Against the forward's kernel (tab_gemm.cuh) two things change.  The operands are split into seven
// 8-bit balanced digits (Digits7x8: 28 digit products per output instead of 45, seven MMAs per 16-deep
// K slice, digit s of A against B's digits 0 .. 6 - s at once, N = 32 (7 - s)), exact while K <= 144.
// And a unit's accumulators (7 diagonals x 32 columns) take 224 TMEM columns, so two of them fit: the
// MMAs of one unit run while the epilogue warps read, recombine and scatter the other's, instead of
// the tensor core waiting for every epilogue.  Roles: warp 0 moves each slice's A and B blocks into a
// ring of five stages (bulk copies counted on the stage's "full" barrier), lane 0 of warp 1 issues the
// MMAs into accumulator buffer (unit & 1) once the epilogue has released it ("tmem_free") and commits
// "acc_full" for that buffer, warp 10 builds each unit's slot table (the run slot of every (interval,
// atom) of the unit, from the atoms' slot keys) and column exponents into table buffer (unit & 1)
// ahead of the epilogue ("tbl_full", released by "tbl_empty"), and eight epilogue warps (two per TMEM
// lane quadrant, 16 columns each) finish the outputs.  (Measured: with the epilogue warps building the
// tables themselves, the tensor core waited for the epilogue about 40 % of the time.)  Every wait is bounded; a wait that gives up stops the CTA's copies and MMAs,
// its remaining outputs are NaN and one timeout is counted (dp_tc_wait_timeouts).
#pragma once

#include "tab_gemm.cuh"
#include "tc_gemm.cuh"

namespace dpc {
namespace {
namespace tb {
using namespace tc;
using tg::wait_or_abort;

constexpr int kSB = Digits7x8::kNS;      // 7 digits of 8 bits
constexpr int kTNB = 32;                 // columns per unit: 8 atoms x 4 (k)
constexpr int kAtomsB = kTNB / 4;
constexpr int kStagesB = 5;
constexpr int kPlaneAB = kTM * kTK * 2;  // one digit plane of a 128-row A block: 4 KB
constexpr int kPlaneBB = kTNB * kTK * 2; // of a 32-row B block: 1 KB
constexpr int kStageBytesB = kSB * (kPlaneAB + kPlaneBB);
constexpr int kMaxKB = 144;              // K (channels, padded to 16) of one exact share
constexpr int kEpiWarpsB = 8;
constexpr int kThreadsB = 32 * (3 + kEpiWarpsB);  // producer, MMA issuer, epilogue, table warp
constexpr int kTableWarp = 2 + kEpiWarpsB;
constexpr int kEpiColsB = kTNB / 2;      // columns per epilogue warp
constexpr uint32_t kBufColsB = 256;      // TMEM columns per accumulator buffer (7 x 32 used)
constexpr int kScatKeysB = kTM / 4 + 1;  // keys a 128-row tile touches (kq >= 4)
static_assert(7ll * 128 * 128 * kMaxKB < (1ll << 24), "exact fp32 diagonal sums");
static_assert(kSB * kTNB <= (int)kBufColsB && 2 * kBufColsB <= kTmemCols, "two accumulator buffers");
static_assert(kStageBytesB % 1024 == 0, "stages stay 1024-byte aligned");

struct Params {
  const unsigned char *aplanes;  // A = C'_alpha: blocks [Mp / 128][ka] of kSB x kPlaneAB bytes
  const int *Eexp;               // [Mp] row exponents
  int ka;                        // K slices: the channels padded to 16, / 16 (<= 9)
  const unsigned char *bplanes;  // B = dT^T of the chunk: blocks [ntiles][ka] of kSB x kPlaneBB bytes
  const int *Fexp;               // [32 ntiles] column exponents
  int64_t Mp;
  double *scat;       // [natoms][cap][24]: the wanted outputs, per run slot, finished to f64
  const short *keys;  // [atom0 + natoms][cap]: each atom's slot keys
  const int *nslots;  // [atom0 + natoms]
  int cap, nkeys, kq;
  const int32_t *atype;
  int64_t natoms, atom0;
  int alpha, ntypes;
  const int *units;   // the launch's units (tile | mt << 16), in any order
  const int *nunits;  // their count (device)
};

__host__ __device__ constexpr int unit_code(int tile, int mt) { return tile | (mt << 16); }

// full[5], empty[5], acc_full[2], tmem_free[2], tbl_full[2], tbl_empty[2]
constexpr size_t kBarOffB = (size_t)kStagesB * kStageBytesB;
constexpr size_t kMiscOffB = kBarOffB + (2 * kStagesB + 8) * 8;   // tmem address, abort flag
constexpr size_t kStabOffB = kMiscOffB + 16;                      // two tables: slots, exponents; flags
constexpr int kTableInts = kScatKeysB * kAtomsB + kTNB;          // one table buffer
constexpr size_t kSmemB = kStabOffB + (2 * kTableInts + 4) * 4;
static_assert(kSmemB <= 227 * 1024, "shared memory per block");

__global__ void __launch_bounds__(kThreadsB, 1) bgemm_kernel(const Params P) {
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + kBarOffB);
  uint64_t *empty = full + kStagesB;
  uint64_t *acc_full = empty + kStagesB;
  uint64_t *tmem_free = acc_full + 2;
  uint64_t *tbl_full = tmem_free + 2;
  uint64_t *tbl_empty = tbl_full + 2;
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(smem + kMiscOffB);
  volatile int *abortf = reinterpret_cast<volatile int *>(smem + kMiscOffB + 4);
  // table buffer b: (key of the unit, atom) -> slot or -1, then the unit's 32 column exponents
  int *tables = reinterpret_cast<int *>(smem + kStabOffB);
  int *uflag = tables + 2 * kTableInts;  // [0]: the unit's accumulators and table are ready
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nunits = *P.nunits;

  if (tid == 0) {
    for (int s = 0; s < kStagesB; ++s) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(full + s)));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(empty + s)));
    }
    for (int b = 0; b < 2; ++b) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(acc_full + b)));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(tmem_free + b)), "r"(kEpiWarpsB));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(tbl_full + b)));
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(tbl_empty + b)), "r"(kEpiWarpsB));
    }
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
    if (lane == 0) {
      int g = 0;  // slices loaded so far by this CTA
      bool ok = true;
      for (int u = blockIdx.x; u < nunits && ok; u += gridDim.x) {
        const int c = P.units[u], tile = c & 0xffff, mt = c >> 16;
        for (int j = 0; j < P.ka; ++j, ++g) {
          const int st = g % kStagesB;
          if (g >= kStagesB && !(ok = wait_or_abort(smem_u32(empty + st), (uint32_t)((g / kStagesB - 1) & 1), abortf)))
            break;
          const unsigned char *asrc = P.aplanes + ((size_t)mt * P.ka + j) * (kSB * kPlaneAB);
          const unsigned char *bsrc = P.bplanes + ((size_t)tile * P.ka + j) * (kSB * kPlaneBB);
          const uint32_t bar = smem_u32(full + st), dst = sbase + st * kStageBytesB;
          asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"((uint32_t)kStageBytesB)
                       : "memory");
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
              "l"(asrc), "r"((uint32_t)(kSB * kPlaneAB)), "r"(bar)
              : "memory");
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                  dst + kSB * kPlaneAB),
              "l"(bsrc), "r"((uint32_t)(kSB * kPlaneBB)), "r"(bar)
              : "memory");
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA issuer: per slice the 28 digit products as 7 MMAs into the unit's buffer, per unit a
    // commit on that buffer's acc_full once they have all completed
    if (lane == 0) {
      int g = 0, li = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < nunits && ok; u += gridDim.x) {
        const int b = li & 1;
        if (li >= 2 && !(ok = wait_or_abort(smem_u32(tmem_free + b), (uint32_t)(((li >> 1) - 1) & 1), abortf))) break;
        asm volatile("tcgen05.fence::after_thread_sync;");
        const uint32_t acc0 = tmem + (uint32_t)b * kBufColsB;
        for (int j = 0; j < P.ka; ++j, ++g) {
          const int st = g % kStagesB;
          if (!(ok = wait_or_abort(smem_u32(full + st), (uint32_t)((g / kStagesB) & 1), abortf))) break;
          asm volatile("tcgen05.fence::after_thread_sync;");
          const uint64_t a0 = smem_desc(sbase + st * kStageBytesB);
          const uint64_t b0 = smem_desc(sbase + st * kStageBytesB + kSB * kPlaneAB);
#pragma unroll
          for (int s = 0; s < kSB; ++s) {
            const uint32_t idesc = kIdescNoN | ((uint32_t)((kTNB * (kSB - s)) >> 3) << 17);
            const uint32_t acc = (j > 0 || s > 0) ? 1u : 0u;  // a unit's first digit product writes every diagonal
            asm volatile(
                "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(acc0 + (uint32_t)(s * kTNB)),
                "l"(a0 + (uint64_t)((s * kPlaneAB) >> 4)), "l"(b0), "r"(idesc), "r"(acc));
          }
          asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
              smem_u32(empty + st)));
        }
        // completes when every MMA issued so far has (also after a wait that gave up)
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(acc_full + b)));
        ++li;
      }
    }
    __syncwarp();
  } else if (warp == kTableWarp) {
    // ---- table warp: each unit's slot table and column exponents into table buffer (unit & 1)
    int li = 0;
    for (int u = blockIdx.x; u < nunits; u += gridDim.x) {
      const int c = P.units[u], tile = c & 0xffff, mt = c >> 16;
      const int b = li & 1;
      if (li >= 2) {
        int wv = 1;
        if (lane == 0) wv = wait_or_abort(smem_u32(tbl_empty + b), (uint32_t)(((li >> 1) - 1) & 1), abortf);
        if (!__shfl_sync(0xffffffffu, wv, 0)) break;
      }
      int *stab = tables + b * kTableInts, *fexp_s = stab + kScatKeysB * kAtomsB;
      const int64_t a_first = (int64_t)tile * kAtomsB;
      const int key0 = (int)((int64_t)mt * kTM / P.kq);
      for (int x = lane; x < kScatKeysB * kAtomsB; x += 32) stab[x] = -1;
      fexp_s[lane] = P.Fexp[(int64_t)tile * kTNB + lane];
      __syncwarp();
      // the slot counts of the unit's atoms (0: past the chunk or not of type alpha), lane al < 8
      int nsl = 0;
      if (lane < kAtomsB) {
        const int64_t a = a_first + lane, i = P.atom0 + a;
        nsl = a < P.natoms && (!P.atype || clampi(P.atype[i], 0, P.ntypes - 1) == P.alpha) ? P.nslots[i] : 0;
      }
      int nmax = nsl;
#pragma unroll
      for (int o = 1; o < kAtomsB; o <<= 1) nmax = max(nmax, __shfl_xor_sync(0xffffffffu, nmax, o));
      nmax = __shfl_sync(0xffffffffu, nmax, 0);  // lanes 0 .. 7 hold the maximum; the loop below is uniform
      // (atom, slot) pairs over the lanes, four slots of an atom per pass so that the key loads overlap
      const short *keys = P.keys + (P.atom0 + a_first) * P.cap;
      for (int s0 = 0; s0 < nmax; s0 += 16) {  // uniform
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const int al = lane >> 2, slot = s0 + 4 * h + (lane & 3);
          const int ns = __shfl_sync(0xffffffffu, nsl, al);
          const int key = slot < ns ? keys[(size_t)al * P.cap + slot] : -1;
          if (key >= key0 && key < key0 + kScatKeysB) stab[(key - key0) * kAtomsB + al] = slot;
        }
      }
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(tbl_full + b)) : "memory");
      ++li;
    }
  } else {
    // ---- epilogue: warps 2 .. 9, TMEM lane quadrant warp % 4, columns 16 ((warp - 2) / 4) .. + 15
    const int et = tid - 64;
    const int q = warp & 3, c_lo = ((warp - 2) / 4) * kEpiColsB;
    const int rl = 32 * q + lane;
    int li = 0;
    for (int u = blockIdx.x; u < nunits; u += gridDim.x) {
      const int c = P.units[u], tile = c & 0xffff, mt = c >> 16;
      const int b = li & 1;
      const int64_t m0 = (int64_t)mt * kTM;
      const int64_t a_first = (int64_t)tile * kAtomsB;  // the unit's first atom in the chunk
      const int *stab = tables + b * kTableInts, *fexp_s = stab + kScatKeysB * kAtomsB;
      const int key0 = (int)(m0 / P.kq);
      if (et == 0)
        uflag[0] = !*abortf && wait_or_abort(smem_u32(tbl_full + b), (uint32_t)((li >> 1) & 1), abortf) &&
                   wait_or_abort(smem_u32(acc_full + b), (uint32_t)((li >> 1) & 1), abortf);
      asm volatile("bar.sync 1, %0;" ::"r"(32 * kEpiWarpsB));  // the table is built and the MMAs done
      const bool ok = uflag[0] != 0;
      asm volatile("tcgen05.fence::after_thread_sync;");
      const int Erow = m0 + rl < P.Mp ? P.Eexp[m0 + rl] : 0;
      const int key = (int)((m0 + rl) / P.kq), qq = (int)(m0 + rl - (int64_t)key * P.kq);
      const int key_l = key - key0;
      const bool row_wanted = qq < 6 && key < P.nkeys;
      const uint32_t trow = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)b * kBufColsB;
      // the warp's 16 columns, four (one atom) at a time: each output's seven diagonals recombined
      // exactly as an integer and rounded once to f64 (diag7_to_f64), only where a row of the warp wants
      // the atom's slot of that interval
#pragma unroll 1
      for (int c0 = 0; c0 < kEpiColsB; c0 += 4) {
        float v[kSB][4];
        if (ok) {  // uniform over the CTA
#pragma unroll
          for (int d = 0; d < kSB; ++d)
            asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
                         : "=f"(v[d][0]), "=f"(v[d][1]), "=f"(v[d][2]), "=f"(v[d][3])
                         : "r"(trow + (uint32_t)(d * kTNB + c_lo + c0)));
          asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
          for (int d = 0; d < kSB; ++d) asm volatile("" : "+f"(v[d][0]), "+f"(v[d][1]), "+f"(v[d][2]), "+f"(v[d][3]));
        }
        const int al = (c_lo + c0) >> 2;
        int64_t at = -1;
        if (row_wanted) {
          const int slot = stab[key_l * kAtomsB + al];
          if (slot >= 0) at = ((a_first + al) * P.cap + slot) * 24 + qq;
        }
        if (!__any_sync(0xffffffffu, at >= 0)) continue;
        double val[4];
        int F[4];
        bool rare = false;
#pragma unroll
        for (int k = 0; k < 4; ++k) F[k] = fexp_s[c_lo + c0 + k];
#pragma unroll
        for (int k = 0; k < 4; ++k) val[k] = diag7_to_f64(v, k, Erow, F[k], rare);
        if (__any_sync(0xffffffffu, rare))  // warp-uniform, and never taken with these operands
#pragma unroll
          for (int k = 0; k < 4; ++k)
            val[k] = output_value_rare(v[0][k], v[1][k], v[2][k], v[3][k], v[4][k], v[5][k], v[6][k], 0.f, 0.f, Erow,
                                       F[k], true);
        if (at >= 0)
#pragma unroll
          for (int k = 0; k < 4; ++k) P.scat[at + 6 * k] = ok ? val[k] : __longlong_as_double(0x7ff8000000000000ll);
      }
      asm volatile("tcgen05.fence::before_thread_sync;");
      __syncwarp();
      if (lane == 0) {
        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(tmem_free + b)) : "memory");
        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(tbl_empty + b)) : "memory");
      }
      ++li;
    }
  }

  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  if (tid == 0 && *abortf) atomicAdd(&g_wait_timeouts, 1u);
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

// One launch over the units of P's list: one CTA per SM (its shared-memory size set on first use per device).
int launch(const Params &P, cudaStream_t st, const char *who) {
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(cudaGetLastError()));
  static std::atomic<unsigned long long> set_on{0};  // bit d: the attribute is set on device d
  if (dev < 64 && !(set_on.load(std::memory_order_acquire) >> dev & 1ull)) {
    const cudaError_t e = cudaFuncSetAttribute(bgemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemB);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
    set_on.fetch_or(1ull << dev, std::memory_order_acq_rel);
  } else if (dev >= 64) {
    const cudaError_t e = cudaFuncSetAttribute(bgemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemB);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
  }
  bgemm_kernel<<<(unsigned)std::max(nsm, 1), kThreadsB, kSmemB, st>>>(P);
  return launch_status(who);
}

}  // namespace tb
}  // namespace
}  // namespace dpc
