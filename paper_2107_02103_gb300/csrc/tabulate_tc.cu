// Tabulated embedding + contraction (Sec. II, kernel fusion) in f64 with the
// per-interval contraction on the tcgen05 tensor cores.
//
// The fused forward is a sum over the valid neighbour rows j of atom i,
//   T_i[k][m] = (1/N_c) sum_j R~_j[k] g_m^l(t_j),  g_m^l(t) = sum_q c_q^{l,m} t^q (q = 0..5),
// l the row's interval and t its offset from the interval's left node.  With
// u = t / Delta_l (Delta_l the interval's step, so 0 <= u <= 1) and the scaled
// coefficients c'_q^{l,m} = c_q^{l,m} Delta_l^q, it regroups per interval into
// moments of the rows that fall in it,
//   W_i[k][(l, q)] = sum_{j in l} R~_j[k] u_j^q,     T_i[k][m] = (1/N_c) sum_{(l, q)} W_i[k][(l, q)] c'_q^{l,m},
// a GEMM whose K index is (neighbour type, interval, power): the same sum as
// the per-row evaluation, associated per interval.  The backward is the
// transposed GEMM, on the unscaled coefficients (its A rows 6 key + q each
// carry their own exponent, so no scale is needed there), and the rows'
// polynomials in t itself:
//   dW_i[k][(l, q)] = (1/N_c) sum_m dT_i[k][m] c_q^{l,m},
//   dE/dR~_j[k] = sum_q dW_i[k][(l, q)] t_j^q,
//   dE/ds_j     = sum_k R~_j[k] sum_{q >= 1} q dW_i[k][(l, q)] t_j^(q-1)   (0 where s_j was clamped).
// The FP64 pipe keeps the per-row work (24 FMAs per row for W, 40 for the
// derivatives); the per-interval work (24 M1 FMAs per interval and atom in
// each direction), which is most of it, runs as exact digit-split GEMMs on
// the tensor cores (tc_gemm.cuh), at f64 accuracy.
//
// K layout, per centre type: key = beta nint + l (neighbour type beta, interval
// l), and column 6 key + q of the GEMM holds power q, so an interval lies in
// one or two 16-deep K slices.  An atom touches only the intervals its
// rows fall in: the W values are stored per run of rows (one slot per
// interval an atom uses, found through a per-atom map), and the GEMMs skip the
// slices (forward) or output tiles (backward) that no atom of a tile uses.
//
// C'_alpha and its digit planes are made once per table by dp_tabulate_tc_plan_f64 (the plan).
// Per chunk of at most kChunkAtoms atoms:
//   forward:  runs_kernel<true> (slot keys, W, column exponents, slice flags), slice_list_kernel (each
//             tile's used slices), fwd_schedule_kernel (every centre type's items cut into pieces of
//             equal cost per CTA), tgemm_kernel<true> (tab_gemm.cuh, one launch; A = C'_alpha^T:
//             channels x K, B = W^T: K x (atom, k), its digit planes made in shared memory from W; an
//             uncut item writes its atoms' T, a piece its exact 128-bit partial sums),
//             fwd_finish_kernel (T of the cut items, and D_i = T_i^T T_i[:, :M2] when asked for);
//   backward: runs_kernel<false> (slot keys, slice flags; skipped when the forward's are reused),
//             the split of dT (B), the GEMM units, and per centre type the GEMM (A = C'_alpha: K x
//             channels, B = dT^T) scattering each used (atom, interval) block to its run slot --
//             bgemm_kernel (tab_gemm_b8.cuh: 8-atom tiles, seven 8-bit digits) when M1 rounds up to
//             at most 144, else tgemm_kernel<false> (12-atom tiles, nine 6-bit digits) -- and
//             rows_kernel (dE/ds, dE/dR~).
// The environment-fused calls (dp_tabulate_fusion_env_*_tc_f64) form each row from coordinates in
// runs_kernel<.., true> and add each row's force and virial in rows_force_kernel instead.
// The slot keys, their counts and the slice flags of every atom stay in the work buffer after
// the forward, so that a backward on the same inputs can skip its own key pass.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "dp_common.cuh"
#include "env_row.cuh"
#include "tab_gemm.cuh"
#include "tab_gemm_b8.cuh"
#include "tc_gemm.cuh"

namespace dpc {
namespace {
namespace tt {
using namespace tc;

constexpr int kQ = 6;                 // K entries per interval: u^0 .. u^5
constexpr int kCols = 4;              // GEMM columns per atom: k = 0 .. 3
constexpr int kTileAtoms = kTN / kCols;  // 12 atoms per 48-column tile
constexpr int64_t kChunkAtoms = 16416;   // a multiple of 24 (12- and 8-atom tiles; 65,664 columns)
constexpr int kShareSlices = kMaxShareSlices;  // used K slices per forward share (112, the exactness bound)
constexpr size_t kPartBudget = (size_t)1 << 30;  // bytes of the forward's partial results per chunk at most
constexpr int kMaxCtasF = 160;  // CTAs of the forward GEMM at most (its part slots are sized for them)
constexpr int kEpiCost = 6;     // a forward unit's epilogue, in slices' time, for the forward schedule
constexpr int kMaxKeys = 4096;  // ntypes x nint: each warp's key map (int16) lives in shared memory
static_assert(kChunkAtoms % kTileAtoms == 0 && kChunkAtoms % 8 == 0, "whole tiles per chunk");

// Sizes shared by the kernels, the plan and the work-buffer layout.
struct Shape {
  int ntypes, nint, nkeys, M1, cap;
  int Kp;    // round_up(6 nkeys, 16): K of the forward GEMM, rows of the backward A
  int nsl;   // Kp / 16
  int Mpf;   // round_up(M1, 128): rows of the forward A
  int Kpm;   // round_up(M1, 16): K of the backward GEMM
  int Mpb;   // round_up(Kp, 128): rows of the backward A
  int64_t nloc, tiles_all;    // atoms of the call and their 12-atom tiles
  int64_t chunk, Np, ntiles;  // atoms per chunk, its columns round_up(4 chunk, 48), Np / 48
  int zmax;                   // forward shares per tile at most
  int64_t maxunits;           // backward GEMM units (9 x 6 digits) per chunk and centre type at most
  int64_t nitems;             // forward items per chunk: (type, 12-atom tile, 128-row tile of A)
  int64_t maxpieces, maxslots;  // forward pieces and part slots per chunk at most
  bool b8;                    // the backward GEMM uses the 7 x 8-bit digits on 8-atom tiles (Kpm <= 144)
  int64_t Np8, ntiles8;       // its columns round_up(4 chunk, 32) and tiles Np8 / 32
  int64_t maxunits8;          // its units per chunk and centre type at most
};

// The plan: C' of every centre type and the digit planes of both GEMMs' A operands.
struct PlanLayout {
  size_t nodes, cp, afwd, efwd, abwd, ebwd, total;
};

// The work buffer: the slot keys, their counts and the slice flags of every atom of the call
// (kept from the forward for the backward), then one chunk's scratch.
struct Layout {
  size_t keys, nslots, occ, map, slist, scount, units, nunits, pieces, pcta, cta_start, npieces, pfirst, fexp, bplanes,
      w, part, total;
};

size_t take(size_t &off, size_t bytes) {
  const size_t at = off;
  off += (size_t)round_up((int64_t)bytes, 256);
  return at;
}

Shape table_shape(const TableGeom &g, int ntypes, int M1) {
  Shape s{};
  s.ntypes = ntypes;
  s.nint = g.nint;
  s.nkeys = ntypes * g.nint;
  s.M1 = M1;
  s.Kp = (int)round_up((int64_t)s.nkeys * kQ, kTK);
  s.nsl = s.Kp / kTK;
  s.Mpf = (int)round_up(M1, kTM);
  s.Kpm = (int)round_up(M1, kTK);
  s.Mpb = (int)round_up(s.Kp, kTM);
  s.zmax = (s.nsl + kShareSlices - 1) / kShareSlices;
  s.b8 = s.Kpm <= tb::kMaxKB;
  return s;
}

Shape make_shape(const TableGeom &g, int64_t nloc, int nnei, int ntypes, int M1) {
  Shape s = table_shape(g, ntypes, M1);
  s.cap = std::min(nnei, s.nkeys);
  s.nloc = nloc;
  s.tiles_all = (nloc + kTileAtoms - 1) / kTileAtoms;
  int64_t chunk = std::min<int64_t>(round_up(std::max<int64_t>(nloc, 1), kTileAtoms), kChunkAtoms);
  // part slots: two per CTA boundary, and every piece of an item whose used slices exceed one share
  auto slots_for = [&](int64_t c) {
    const int64_t items = (int64_t)s.ntypes * (round_up(kCols * c, kTN) / kTN) * (s.Mpf / kTM);
    return 2 * kMaxCtasF + (s.zmax > 1 ? items * s.zmax : 0);
  };
  while (chunk > kTileAtoms && (size_t)slots_for(chunk) * s.Mpf * kTN * sizeof(float4) > kPartBudget)
    chunk = round_up(chunk / 2, kTileAtoms);
  s.chunk = chunk;
  s.Np = round_up(kCols * chunk, kTN);
  s.ntiles = s.Np / kTN;
  s.maxunits = s.ntiles * (s.Mpb / kTM);
  s.nitems = (int64_t)s.ntypes * s.ntiles * (s.Mpf / kTM);
  s.maxpieces = s.nitems * s.zmax + kMaxCtasF;
  s.maxslots = slots_for(chunk);
  s.Np8 = round_up(kCols * chunk, tb::kTNB);
  s.ntiles8 = s.Np8 / tb::kTNB;
  s.maxunits8 = s.ntiles8 * (s.Mpb / kTM);
  return s;
}

PlanLayout plan_layout(const Shape &s) {
  PlanLayout L{};
  size_t off = 0;
  const size_t nt = (size_t)s.ntypes;
  L.nodes = take(off, (size_t)(s.nint + 1) * sizeof(double));
  L.cp = take(off, nt * s.Kp * s.M1 * sizeof(double));
  L.afwd = take(off, nt * kS * (size_t)s.Mpf * s.Kp * 2);
  L.efwd = take(off, nt * s.Mpf * sizeof(int));
  L.abwd = take(off, nt * (s.b8 ? tb::kSB : kS) * (size_t)s.Mpb * s.Kpm * 2);
  L.ebwd = take(off, nt * s.Mpb * sizeof(int));
  L.total = off;
  return L;
}

Layout make_layout(const Shape &s) {
  Layout L{};
  size_t off = 0;
  L.keys = take(off, (size_t)std::max<int64_t>(s.nloc, 1) * s.cap * sizeof(short));
  L.nslots = take(off, (size_t)std::max<int64_t>(s.nloc, 1) * sizeof(int));
  L.occ = take(off, (size_t)s.ntypes * std::max<int64_t>(s.tiles_all, 1) * s.nsl);
  L.map = take(off, (size_t)s.chunk * s.nkeys * sizeof(int));
  L.slist = take(off, (size_t)s.ntypes * s.ntiles * s.nsl * sizeof(short));
  L.scount = take(off, (size_t)s.ntypes * s.ntiles * sizeof(int));
  L.units = take(off, (size_t)s.ntypes * std::max(s.maxunits, s.maxunits8) * sizeof(int));
  L.nunits = take(off, (size_t)s.ntypes * sizeof(int));
  L.pieces = take(off, (size_t)s.maxpieces * sizeof(int4));
  L.pcta = take(off, (size_t)s.maxpieces * sizeof(int));
  L.cta_start = take(off, (size_t)(kMaxCtasF + 1) * sizeof(int));
  L.npieces = take(off, (size_t)s.nitems * sizeof(int));
  L.pfirst = take(off, (size_t)s.nitems * sizeof(int));
  L.fexp = take(off, (size_t)std::max(s.Np, s.Np8) * sizeof(int));
  L.bplanes = take(off, s.b8 ? (size_t)s.ntiles8 * (s.Kpm / kTK) * tb::kSB * tb::kPlaneBB  // the backward's dT planes
                             : (size_t)s.ntiles * (s.Kpm / kTK) * kS * kPlaneB);
  L.w = take(off, (size_t)s.chunk * s.cap * 24 * sizeof(double));  // moments (forward) or their gradients
  L.part = take(off, (size_t)s.maxslots * s.Mpf * kTN * sizeof(longlong2));
  L.total = off;
  return L;
}

// C'[alpha][6 key + q][m] = c_q Delta_l^q / N_c (key = beta nint + l; rows past the keys: 0).
// The interval's block of the table is pair-planar [3][M1][2] holding (a, b, c, d, e, f), the
// coefficients of t^5 .. t^0.
// kU: the coefficients of u^q, c_q Delta^q (the forward's); else of t^q, c_q (the backward's)
__global__ void __launch_bounds__(256) coef_kernel(const double *__restrict__ table, TableGeom g, int ntypes, int M1,
                                                   int Kp, double scale, bool kU, double *__restrict__ Cp) {
  const int64_t total = (int64_t)ntypes * Kp * M1;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total; x += (int64_t)gridDim.x * blockDim.x) {
    const int m = (int)(x % M1);
    const int64_t rest = x / M1;
    const int r = (int)(rest % Kp), alpha = (int)(rest / Kp);
    const int key = r / kQ, q = r - kQ * key;
    double v = 0.0;
    if (key < ntypes * g.nint) {
      const int beta = key / g.nint, l = key - beta * g.nint;
      const double *blk = table + ((size_t)(alpha * ntypes + beta) * g.nint + l) * M1 * 6;
      const int j = 5 - q;  // position of t^q's coefficient in (a .. f)
      const double c = blk[(size_t)(j >> 1) * 2 * M1 + 2 * m + (j & 1)];
      const double delta = l < g.n0 ? g.stride0 : g.stride1;
      double p = 1.0;
      if (kU)
        for (int e = 0; e < q; ++e) p *= delta;
      v = c * p * scale;
    }
    Cp[x] = v;
  }
}

// The grid's nodes x_0 .. x_nint as the interval search forms them (node_x), for the per-row kernels.
__global__ void nodes_kernel(TableGeom g, double *__restrict__ nodes) {
  for (int l = blockIdx.x * blockDim.x + threadIdx.x; l <= g.nint; l += gridDim.x * blockDim.x) nodes[l] = node_x(g, l);
}

// An f32 value within 2^-23 (relative) of s, formed from the fields of s by integer operations (no
// FP64 instruction); ok is false where that fails: |s| outside [2^-100, 2^100), zero, inf, NaN.
__device__ __forceinline__ float approx_f32(double s, bool &ok) {
  const unsigned hi = (unsigned)__double2hiint(s), lo = (unsigned)__double2loint(s);
  const int e = (int)((hi >> 20) & 0x7ff) - 1023;
  ok = e > -100 && e < 100;
  return __uint_as_float((hi & 0x80000000u) | ((unsigned)(e + 127) << 23) | ((hi & 0xfffffu) << 3) | (lo >> 29));
}

// floor(x) clamped into [0, n], for x below 2^22, on the FP32 pipe: 2^23 added with rounding down.
__device__ __forceinline__ int floor_clamped(float x, int n) {
  return __float_as_int(__fadd_rd(fminf(fmaxf(x, 0.0f), (float)n), 8388608.0f)) - 0x4B000000;
}

// The interval search of the tensor-core path's per-row kernels.  The segment and the index come from
// the f32 approximation of s; t = s - x_l is one f64 subtraction from the node table.  The f32 index can
// differ from floor((s - x_0) / Delta) by one where s lies within ~1e-4 steps of a node; either interval
// is correct there (the table is C2, so both polynomials agree to the rounding at the node, and t then
// lies a hair outside [0, Delta]).  Inputs within 2^-18 (relative) of lower, upper or upper_ext, where
// the f32 comparison could take the wrong side, and inputs outside the f32 range take the f64 search,
// whose clamping they follow exactly.  Deterministic: the forward and the backward find the same l.
__device__ __forceinline__ int locate_fast(const TableGeom &g, const TableGeomF &f, const double *__restrict__ nodes,
                                           double s, double &t, bool &clamped) {
  bool ok;
  const float sf = approx_f32(s, ok);
  const float tol = 0x1p-18f * fabsf(sf);
  if (!ok || fabsf(sf - f.lower) <= tol || fabsf(sf - f.upper) <= tol || fabsf(sf - f.upper_ext) <= tol)
    return locate(g, s, t, clamped);
  clamped = sf < f.lower || sf >= f.upper_ext;
  if (sf < f.lower) {
    t = 0.0;
    return 0;
  }
  if (sf >= f.upper_ext) {
    t = g.n1 > 0 ? g.stride1 : g.stride0;
    return g.nint - 1;
  }
  const int l = sf < f.upper ? floor_clamped((sf - f.lower) * f.inv0, g.n0 - 1)
                             : g.n0 + floor_clamped((sf - f.upper) * f.inv1, g.n1 - 1);
  t = s - __ldg(nodes + l);
  return l;
}

// The environment matrix's inputs, where the tensor-core path forms its rows from coordinates itself
// (dp_tabulate_fusion_env_*_tc_f64: s and R~ never reach HBM, nor ds and dR~ in the backward).
struct EnvRow {
  const double *coord;   // [nall][3]
  const int32_t *nlist;  // [nloc][nnei]: the neighbour's index into coord, or -1 (each segment's first)
  double rcs, rc, inv_width, mean, inv_std, inv_std_all;
  int kind;
};

// Row (i, j) as dp_env_mat forms it, by the same operations: d = x_j - x_i, r, 1/r, s(r) and ds/dr, the
// table input and R~[0] sh = (s - mean)/std, and R~[1 .. 3] = s d / (r std_all).
struct EnvVals {
  double d[3], inv_r, sv, dsv, r4[4];
};
__device__ __forceinline__ EnvVals env_vals(const EnvRow &E, int64_t i, int j) {
  EnvVals v;
  const double xi = E.coord[3 * i], yi = E.coord[3 * i + 1], zi = E.coord[3 * i + 2];
  v.d[0] = E.coord[3 * (int64_t)j] - xi;
  v.d[1] = E.coord[3 * (int64_t)j + 1] - yi;
  v.d[2] = E.coord[3 * (int64_t)j + 2] - zi;
  const double r2 = fma(v.d[0], v.d[0], fma(v.d[1], v.d[1], v.d[2] * v.d[2]));
  const double r = sqrt(r2);
  v.inv_r = recip(r);
  weight(E, r, v.inv_r, v.sv, v.dsv);
  const double a = v.sv * v.inv_r * E.inv_std_all;
  v.r4[0] = (v.sv - E.mean) * E.inv_std;
  v.r4[1] = a * v.d[0];
  v.r4[2] = a * v.d[1];
  v.r4[3] = a * v.d[2];
  return v;
}

// Valid rows per type segment of atom i from its neighbour list (the rows with a neighbour, each
// segment's first, as dp_env_mat counts them) into nvb, and into nvalid_out when given; their total.
__device__ __forceinline__ int env_valid_rows(const EnvRow &E, int nnei, const int *sel, int ntypes, int64_t i,
                                              int lane, int *nvb, int32_t *nvalid_out) {
  int count = 0;  // lane b < ntypes: segment b's rows with a neighbour
  for (int q0 = 0; q0 < nnei; q0 += 32) {  // uniform
    const int q = q0 + lane;
    const int j = q < nnei ? __ldg(E.nlist + i * nnei + q) : -1;
    int b = 0, lim = sel[0];
#pragma unroll
    for (int c = 1; c < DP_MAX_TYPES; ++c)
      if (c < ntypes && q >= lim) {
        b = c;
        lim += sel[c];
      }
#pragma unroll
    for (int c = 0; c < DP_MAX_TYPES; ++c) {
      if (c >= ntypes) break;  // uniform
      const int n = __popc(__ballot_sync(0xffffffffu, j >= 0 && b == c));
      if (lane == c) count += n;
    }
  }
  if (lane < DP_MAX_TYPES) nvb[lane] = lane < ntypes ? count : 0;
  if (nvalid_out && lane < ntypes) nvalid_out[i * ntypes + lane] = count;
  __syncwarp();
  int nv = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q) nv += nvb[q];
  return nv;
}

struct RunsParams {
  const double *s, *Rt;
  EnvRow env;           // kEnv: rows from coordinates (s and Rt unused)
  int32_t *nvalid_out;  // kEnv forward: the counts of valid rows it finds
  const int32_t *nvalid, *atype;
  TableGeom g;
  TableGeomF gf;
  const double *nodes;  // [nint + 1] (the plan's)
  int64_t atom0, natoms, tiles_all;  // the chunk's first atom (a multiple of 12) and size; all tiles
  int nnei, ntypes, nkeys, cap, nsl;
  int sel[DP_MAX_TYPES];
  short *keys;         // [nloc][cap]: key of each slot (every atom of the call)
  int *nslots;         // [nloc]: slots in use
  unsigned char *occ;  // [ntypes][tiles_all][nsl]: the K slices some atom of the tile uses
  int *map;            // forward: [natoms][nkeys] run slot of the key, or -1 (this chunk)
  double *W;           // forward: [natoms][cap][24] moments W[k][q] at 6 k + q
  int *fexp;           // forward: [Np] exponents of the columns 4 a + k
};

struct alignas(16) RunsStage {
  double r[32][4];
  double tp[32][6];
  int key[32];
  int nvb[DP_MAX_TYPES];
};

// Valid rows per type segment of atom i (clamped into [0, sel]) into nvb; returns their total.
__device__ __forceinline__ int valid_rows(const int32_t *nvalid, const int *sel, int ntypes, int64_t i, int lane,
                                          int *nvb) {
  int sl = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q)
    if (lane == q) sl = sel[q];
  int x = 0;
  if (lane < ntypes) x = clampi(nvalid ? __ldg(nvalid + i * ntypes + lane) : sl, 0, sl);
  if (lane < DP_MAX_TYPES) nvb[lane] = x;
  __syncwarp();
  int nv = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q) nv += nvb[q];
  return nv;
}

// Row index of valid row v (type segments in order, the valid rows of each first) and its segment.
__device__ __forceinline__ int valid_row(int v, const int *nvb, const int *sel, int ntypes, int &b) {
  int cum = 0, lim = nvb[0], off = 0;
  b = 0;
#pragma unroll
  for (int q = 1; q < DP_MAX_TYPES; ++q)
    if (q < ntypes && v >= lim) {
      b = q;
      cum = lim;
      lim += nvb[q];
      off += sel[q - 1];
    }
  return off + (v - cum);
}

// One warp per atom: the runs of rows sharing an interval (consecutive rows with one key; rows
// sorted by distance give one run per interval, and a key met again adds to its slot), each
// interval's slot (a shared-memory map of the keys; each slot's key and the slot count are written
// out) and the flags of its K slices for the atom's tile; forward also the map, its moments W and
// the atom's four column exponents (over every value written, which bounds the final ones).
// Warps (one atom each) per block of the runs and rows kernels: a few per block, so that launching
// thousands of tiny blocks does not set the pace of a short kernel.
constexpr int kRunsWarps = 4, kRowsWarps = 4;

template <bool kMom, bool kEnv = false>
__global__ void __launch_bounds__(32 * kRunsWarps) runs_kernel(const RunsParams P) {
  __shared__ RunsStage stw[kRunsWarps];
  extern __shared__ short smapw[];  // [kRunsWarps][nkeys]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t a = (int64_t)blockIdx.x * kRunsWarps + warp;
  if (a >= P.natoms) return;  // warp-uniform
  RunsStage &st = stw[warp];
  short *smap = smapw + (size_t)warp * P.nkeys;
  const int64_t i = P.atom0 + a;
  for (int k = lane; k < P.nkeys; k += 32) smap[k] = -1;
  const int nv = kEnv ? env_valid_rows(P.env, P.nnei, P.sel, P.ntypes, i, lane, st.nvb, P.nvalid_out)
                      : valid_rows(P.nvalid, P.sel, P.ntypes, i, lane, st.nvb);  // (their __syncwarp orders the reset)
  const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
  unsigned char *occ = P.occ + ((size_t)alpha * P.tiles_all + (size_t)(i / kTileAtoms)) * P.nsl;
  short *keys = P.keys + i * P.cap;
  double *Wa = kMom ? P.W + (size_t)a * P.cap * 24 : nullptr;
  int nslot = 0;
  int cur = -1;       // key of the open run (uniform)
  double wv = 0.0;    // its moment W[k][q] on lane 6 k + q < 24
  int eb = 0;         // largest exponent field written by this lane
  auto flush = [&]() {  // uniform
    int slot = smap[cur];
    const bool fresh = slot < 0;
    __syncwarp();
    if (fresh) {
      slot = nslot++;
      if (lane == 0) {
        smap[cur] = (short)slot;
        keys[slot] = (short)cur;
        occ[kQ * cur / kTK] = 1;  // the key's entries 6 key .. 6 key + 5, in one or two slices
        occ[(kQ * cur + kQ - 1) / kTK] = 1;
      }
    }
    if (kMom && lane < 24) {
      double *w = Wa + (size_t)slot * 24 + lane;
      const double x = fresh ? wv : *w + wv;
      *w = x;
      eb = max(eb, exp_bits(x));
    }
    __syncwarp();
  };
  const double *srow = P.s + i * P.nnei;
  const double *Rrow = P.Rt + i * P.nnei * 4;
  for (int base = 0; base < nv; base += 32) {
    const int v = base + lane;
    if (v < nv) {
      int b;
      const int row = valid_row(v, st.nvb, P.sel, P.ntypes, b);
      double t, sv, r4[4];
      if constexpr (kEnv) {
        const EnvVals ev = env_vals(P.env, i, __ldg(P.env.nlist + i * P.nnei + row));
        sv = ev.r4[0];
#pragma unroll
        for (int k = 0; k < 4; ++k) r4[k] = ev.r4[k];
      } else {
        sv = __ldg(srow + row);
      }
      bool clamped;
      const int l = locate_fast(P.g, P.gf, P.nodes, sv, t, clamped);
      st.key[lane] = b * P.g.nint + l;
      if constexpr (kMom) {
        Vec4<double> rr;
        if constexpr (kEnv)
          rr = Vec4<double>{r4[0], r4[1], r4[2], r4[3]};
        else
          rr = ld4(Rrow + (size_t)row * 4);
        st.r[lane][0] = rr.x;
        st.r[lane][1] = rr.y;
        st.r[lane][2] = rr.z;
        st.r[lane][3] = rr.w;
        const double u = t * (l < P.g.n0 ? P.g.inv0 : P.g.inv1);
        const double u2 = u * u, u3 = u2 * u;
        st.tp[lane][0] = 1.0;
        st.tp[lane][1] = u;
        st.tp[lane][2] = u2;
        st.tp[lane][3] = u3;
        st.tp[lane][4] = u2 * u2;
        st.tp[lane][5] = u3 * u2;
      }
    }
    __syncwarp();
    const int cnt = min(32, nv - base);
    const int mykey = lane < cnt ? st.key[lane] : -1;
    const int prev = __shfl_up_sync(0xffffffffu, mykey, 1);
    unsigned starts = __ballot_sync(0xffffffffu, lane < cnt && (lane == 0 || mykey != prev));
    while (starts) {  // uniform, run by run
      const int u0 = __ffs(starts) - 1;
      starts &= starts - 1;
      const int e = starts ? __ffs(starts) - 1 : cnt;
      const int key = __shfl_sync(0xffffffffu, mykey, u0);
      if (key != cur) {
        if (cur >= 0) flush();
        cur = key;
        wv = 0.0;
      }
      if (kMom && lane < 24) {
        const int k = lane / 6, q = lane - 6 * (lane / 6);
        for (int j = u0; j < e; ++j) wv = fma(st.r[j][k], st.tp[j][q], wv);
      }
    }
    __syncwarp();
  }
  if (cur >= 0) flush();
  if (lane == 0) P.nslots[i] = nslot;
  if constexpr (kMom) {
    int *map = P.map + a * P.nkeys;
    for (int k = lane; k < P.nkeys; k += 32) map[k] = smap[k];
    int m = eb;  // per k: the largest over its six lanes
#pragma unroll
    for (int q = 1; q < 6; ++q) m = max(m, __shfl_sync(0xffffffffu, eb, min(lane + q, 31)));
    if (lane < 24 && lane % 6 == 0) P.fexp[kCols * a + lane / 6] = exp_of_max(m);
  }
}

// The used K slices of each tile of the chunk, in order, and their count, per centre type (one warp per
// (type, tile)).
__global__ void __launch_bounds__(128) slice_list_kernel(const unsigned char *__restrict__ occ, int64_t tiles_all,
                                                         int64_t tile0, int64_t ntiles, int ntypes, int nsl,
                                                         short *__restrict__ list, int *__restrict__ count) {
  const int lane = threadIdx.x & 31;
  const int64_t w = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  if (w >= (int64_t)ntypes * ntiles) return;  // warp-uniform
  const int t = (int)(w / ntiles);
  const int64_t tile = w - (int64_t)t * ntiles;
  const unsigned char *f = occ + ((size_t)t * tiles_all + tile0 + tile) * nsl;
  short *out = list + ((size_t)t * ntiles + tile) * nsl;
  int rank = 0;
  for (int b = 0; b < nsl; b += 32) {  // uniform
    const bool used = b + lane < nsl && f[b + lane] != 0;
    const unsigned m = __ballot_sync(0xffffffffu, used);
    if (used) out[rank + __popc(m & ((1u << lane) - 1u))] = (short)(b + lane);
    rank += __popc(m);
  }
  if (lane == 0) count[(size_t)t * ntiles + tile] = rank;
}

// Exclusive prefix sum over a block of 1024 threads of one value per thread; the block's total in *total.
__device__ long long block_scan_1024(long long v, long long *red, long long *total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  long long x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) red[wid] = x;
  __syncthreads();
  if (wid == 0) {
    long long z = red[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, z, o);
      if (lane >= o) z += y;
    }
    red[lane] = z;  // inclusive over the warps
  }
  __syncthreads();
  const long long before = (wid ? red[wid - 1] : 0ll) + x - v;
  *total = red[31];
  __syncthreads();  // red is reused by the next scan
  return before;
}

// The forward GEMM's schedule over one chunk: every item (type, tile, 128-row tile of A) with used slices
// costs its slice count plus kEpiCost; CTA b takes the cost range [b R, (b + 1) R) of the items' running
// sum, R = ceil(total / ncta), so that every CTA gets the same work.  An item is cut where a CTA's range
// begins and every 112 slices (the exactness bound of a share); the pieces of a cut item write their
// partial results to consecutive part slots, which fwd_finish_kernel sums.  One block of 1024 threads,
// each over a run of consecutive items.
__global__ void __launch_bounds__(1024) fwd_schedule_kernel(const int *__restrict__ scount, int64_t nitems,
                                                            int64_t ntiles, int nmt, int ncta, int4 *__restrict__ pieces,
                                                            int *__restrict__ pcta, int *__restrict__ cta_start,
                                                            int *__restrict__ npieces, int *__restrict__ pfirst) {
  __shared__ long long red[32];
  __shared__ long long s_R;
  const int64_t per = (nitems + 1023) / 1024;
  const int64_t i0 = min(nitems, (int64_t)threadIdx.x * per), i1 = min(nitems, i0 + per);
  auto ns_of = [&](int64_t it) { return scount[it / nmt]; };  // item (t ntiles + tile) nmt + mt
  long long c = 0;
  for (int64_t it = i0; it < i1; ++it) {
    const int ns = ns_of(it);
    c += ns > 0 ? ns + kEpiCost : 0;
  }
  long long total;
  const long long P0 = block_scan_1024(c, red, &total);
  if (threadIdx.x == 0) s_R = max(1ll, (total + ncta - 1) / ncta);
  __syncthreads();
  const long long R = s_R;
  // the pieces of an item: cut where P + x reaches a multiple of R and where x reaches a multiple of 112
  auto for_pieces = [&](long long P, int ns, auto &&f) {
    for (int x = 0; x < ns;) {
      const long long nr = ((P + x) / R + 1) * R - P;
      const int e = (int)min((long long)ns, min(nr, (long long)((x / kShareSlices + 1) * kShareSlices)));
      f(x, e - x, (int)min((P + x) / R, (long long)ncta - 1));
      x = e;
    }
  };
  long long np = 0, nslot = 0, P = P0;
  for (int64_t it = i0; it < i1; ++it) {
    const int ns = ns_of(it);
    int n = 0;
    for_pieces(P, ns, [&](int, int, int) { ++n; });
    np += n;
    nslot += n > 1 ? n : 0;
    P += ns > 0 ? ns + kEpiCost : 0;
  }
  long long np_total, nslot_total;
  long long pbase = block_scan_1024(np, red, &np_total);
  long long sbase = block_scan_1024(nslot, red, &nslot_total);
  P = P0;
  for (int64_t it = i0; it < i1; ++it) {
    const int ns = ns_of(it);
    int n = 0;
    for_pieces(P, ns, [&](int, int, int) { ++n; });
    npieces[it] = n;
    pfirst[it] = n > 1 ? (int)sbase : -1;
    const int64_t tt = it / nmt;
    const int mt = (int)(it - tt * nmt), t = (int)(tt / ntiles), tile = (int)(tt - (int64_t)t * ntiles);
    for_pieces(P, ns, [&](int x, int len, int cta) {
      // tile, (type | mt << 4 | slices << 8), first slice in the tile's list, part slot
      pieces[pbase] = make_int4(tile, t | mt << 4 | len << 8, x, n > 1 ? (int)sbase++ : -1);
      pcta[pbase++] = cta;
    });
    P += ns > 0 ? ns + kEpiCost : 0;
  }
  __syncthreads();
  // CTA b's pieces start at the first piece of a CTA >= b (pieces come in CTA order)
  for (long long i = threadIdx.x; i < np_total; i += blockDim.x) {
    const int cb = pcta[i], ca = i > 0 ? pcta[i - 1] : -1;
    for (int b = ca + 1; b <= cb; ++b) cta_start[b] = (int)i;
  }
  if (threadIdx.x == 0) {
    const int last = np_total > 0 ? pcta[np_total - 1] : -1;
    for (int b = last + 1; b <= ncta; ++b) cta_start[b] = (int)np_total;
  }
}

// The backward GEMM's units: the (tile, 128-row output tile) pairs whose K slices some atom of the tile
// uses, per centre type (one thread per (type, tile)).
__global__ void __launch_bounds__(128) bwd_units_kernel(const unsigned char *__restrict__ occ, int64_t tiles_all,
                                                        int64_t tile0, int64_t ntiles, int ntypes, int nsl, int nmt,
                                                        int64_t maxunits, int *__restrict__ units,
                                                        int *__restrict__ nunits) {
  const int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= (int64_t)ntypes * ntiles) return;
  const int t = (int)(x / ntiles);
  const int64_t tile = x - (int64_t)t * ntiles;
  const unsigned char *f = occ + ((size_t)t * tiles_all + tile0 + tile) * nsl;
  constexpr int kPer = kTM / kTK;  // K slices per 128-row output tile
  for (int mt = 0; mt < nmt; ++mt) {
    bool any = false;
    for (int q = mt * kPer; q < min(nsl, mt * kPer + kPer); ++q) any |= f[q] != 0;
    if (any) units[(size_t)t * maxunits + atomicAdd(nunits + t, 1)] = tg::unit_code((int)tile, mt, 0);
  }
}

// The 7 x 8-bit backward GEMM's units: the (8-atom tile, 128-row output tile) pairs that hold the slot
// of some atom of the tile of type t, from the atoms' slot keys (a key's rows are 6 key .. 6 key + 5),
// per centre type; one block per (type, tile), a warp per atom, the row tiles marked in a shared-memory
// bit set.
constexpr int kMaxRowTiles = 256;
static_assert((int64_t)kMaxKeys * kQ <= (int64_t)kMaxRowTiles * kTM, "row tiles of the backward A fit the bit set");
__global__ void __launch_bounds__(32 * tb::kAtomsB) bwd_units8_kernel(const short *__restrict__ keys,
                                                                    const int *__restrict__ nslots,
                                                                    const int32_t *__restrict__ atype, int ntypes,
                                                                    int cap, int64_t atom0, int64_t natoms,
                                                                    int64_t ntiles8, int64_t maxunits8,
                                                                    int *__restrict__ units, int *__restrict__ nunits) {
  __shared__ unsigned bits[kMaxRowTiles / 32];
  const int lane = threadIdx.x & 31, al = threadIdx.x >> 5;
  const int t = (int)(blockIdx.x / ntiles8);
  const int64_t tile = blockIdx.x - (int64_t)t * ntiles8;
  if (threadIdx.x < kMaxRowTiles / 32) bits[threadIdx.x] = 0u;
  __syncthreads();
  const int64_t a = tile * tb::kAtomsB + al, i = atom0 + a;
  if (a < natoms && (!atype || clampi(atype[i], 0, ntypes - 1) == t)) {  // warp-uniform
    const int ns = nslots[i];
    for (int slot = lane; slot < ns; slot += 32) {
      const int r0 = kQ * (int)keys[i * cap + slot], m_lo = r0 / kTM, m_hi = (r0 + kQ - 1) / kTM;
      atomicOr(&bits[m_lo >> 5], 1u << (m_lo & 31));
      atomicOr(&bits[m_hi >> 5], 1u << (m_hi & 31));
    }
  }
  __syncthreads();
  if (al != 0) return;
  const unsigned word = lane < kMaxRowTiles / 32 ? bits[lane] : 0u;
  const int cnt = __popc(word);
  int before = cnt;  // inclusive prefix over the lanes
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, before, o);
    if (lane >= o) before += y;
  }
  const int total = __shfl_sync(0xffffffffu, before, 31);
  int base = 0;
  if (lane == 0 && total) base = atomicAdd(nunits + t, total);
  base = __shfl_sync(0xffffffffu, base, 0) + before - cnt;
  for (unsigned m = word; m; m &= m - 1u)
    units[(size_t)t * maxunits8 + base++] = tb::unit_code((int)tile, 32 * lane + __ffs((int)m) - 1);
}

// The forward's finish, one block per atom of the chunk: T of an atom whose item (its centre type, its
// tile, a 128-row tile of A) was cut into several pieces -- the pieces' exact integers added as 128-bit
// integers and rounded once to f64 (s128_to_f64: no FP64 instruction) -- or has no used slices (T = 0);
// the other atoms' T the GEMM wrote.  Then, when D is wanted, the atom's descriptor D[m][n] =
// sum_k T[k][m] T[k][n] (n < M2) from its T staged in shared memory, in descriptor_kernel's order of
// operations, so that the two give the same bits.
__global__ void __launch_bounds__(128) fwd_finish_kernel(const longlong2 *__restrict__ part, int Mp,
                                                         const int *__restrict__ eexp, const int *__restrict__ fexp,
                                                         const int *__restrict__ npieces,
                                                         const int *__restrict__ pfirst, int64_t ntiles, int nmt,
                                                         int64_t atom0, const int32_t *__restrict__ atype,
                                                         int ntypes, int M1, double *__restrict__ T, int M2,
                                                         double *__restrict__ D) {
  extern __shared__ double Ts[];  // [4][M1], when D is wanted
  const int64_t a = blockIdx.x;
  const int64_t tile = a / kTileAtoms;
  const int al = (int)(a - tile * kTileAtoms);
  const int t = atype ? clampi(atype[atom0 + a], 0, ntypes - 1) : 0;
  const int64_t item0 = ((int64_t)t * ntiles + tile) * nmt;
  bool direct = true;
  for (int mt = 0; mt < nmt; ++mt) direct = direct && npieces[item0 + mt] == 1;
  if (direct && !D) return;  // uniform
  double *Ta = T + (atom0 + a) * kCols * M1;
  for (int e = threadIdx.x; e < kCols * M1; e += blockDim.x) {
    const int k = e / M1, m = e - k * M1, col = al * kCols + k;
    const int np = npieces[item0 + m / kTM];
    double v;
    if (np == 1) {
      v = Ta[e];  // written by the GEMM (read only for D)
    } else {
      const int first = pfirst[item0 + m / kTM];
      long long hi = 0;
      unsigned long long lo = 0;
      bool nan = false;
      for (int z = 0; z < np; ++z) {  // np == 0: a tile without used slices, whose atoms have no valid rows
        const longlong2 x = part[((size_t)(first + z) * kTN + col) * Mp + m];
        const unsigned long long l = lo + (unsigned long long)x.x;
        hi += x.y + (l < lo ? 1 : 0);
        lo = l;
        nan = nan || x.y == tg::kPartNaN;
      }
      bool rare = false;
      const int E = eexp[(size_t)t * Mp + m], F = fexp[tile * kTN + col];
      v = s128_to_f64<kOutExp>(hi, lo, E, F, rare);
      if (rare) v = output_value((__int128)(((unsigned __int128)(unsigned long long)hi << 64) | lo), E, F);
      if (nan) v = __longlong_as_double(0x7ff8000000000000ll);
      Ta[e] = v;
    }
    if (D) Ts[e] = v;
  }
  if (!D) return;  // uniform
  __syncthreads();
  double *Da = D + (atom0 + a) * (int64_t)M1 * M2;
  for (int e = threadIdx.x; e < M1 * M2; e += blockDim.x) {
    const int m = e / M2, n = e - m * M2;
    double v = Ts[m] * Ts[n];
    v = fma(Ts[M1 + m], Ts[M1 + n], v);
    v = fma(Ts[2 * M1 + m], Ts[2 * M1 + n], v);
    v = fma(Ts[3 * M1 + m], Ts[3 * M1 + n], v);
    Da[e] = v;
  }
}

struct RowsParams {
  const double *s, *Rt;
  const int32_t *nvalid, *atype;
  TableGeom g;
  TableGeomF gf;
  const double *nodes;  // [nint + 1] (the plan's)
  int64_t atom0;
  int nnei, ntypes, nkeys, cap;
  int sel[DP_MAX_TYPES];
  const short *keys;   // [nloc][cap]: key of each slot
  const int *nslots;   // [nloc]
  const double *dW;    // [natoms][cap][24]: the backward GEMM's result per slot, dW[k][q] at 6 k + q
  double *ds, *dRt;
  int64_t natoms;
  EnvRow env;             // rows_force_kernel: rows from coordinates,
  double *F, *virial;     // and the forces [nall][3] and virial [9] they add to
};

// One warp per atom, a lane per valid row: the row's interval from s, its run slot from the atom's key map
// (shared memory), the slot's gradient coefficients dW[k][q] read through L1 (the rows of a run share
// them), and dE/dR~ and dE/ds by Horner's rule in u with its derivative; padded rows get zeros.
__global__ void __launch_bounds__(32 * kRowsWarps) rows_kernel(const RowsParams P) {
  __shared__ int nvbw[kRowsWarps][DP_MAX_TYPES];
  extern __shared__ short smapw[];  // [kRowsWarps][nkeys]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t a = (int64_t)blockIdx.x * kRowsWarps + warp;
  if (a >= P.natoms) return;  // warp-uniform
  int *nvb = nvbw[warp];
  short *smap = smapw + (size_t)warp * P.nkeys;
  const int64_t i = P.atom0 + a;
  const short *keys = P.keys + i * P.cap;
  const int nslot = P.nslots[i];
  for (int k = lane; k < P.nkeys; k += 32) smap[k] = -1;
  __syncwarp();
  for (int x = lane; x < nslot; x += 32) smap[keys[x]] = (short)x;  // the map of the atom's keys
  const int nv = valid_rows(P.nvalid, P.sel, P.ntypes, i, lane, nvb);  // (its __syncwarp orders the map)
  const double *dWa = P.dW + (size_t)a * P.cap * 24;
  const double *srow = P.s + i * P.nnei;
  const double *Rrow = P.Rt + i * P.nnei * 4;
  double *dsrow = P.ds + i * P.nnei;
  double *drow = P.dRt + i * P.nnei * 4;
  for (int v = lane; v < nv; v += 32) {
    int b;
    const int row = valid_row(v, nvb, P.sel, P.ntypes, b);
    double t;
    bool clamped;
    const int l = locate_fast(P.g, P.gf, P.nodes, __ldg(srow + row), t, clamped);
    const Vec4<double> rr = ld4(Rrow + (size_t)row * 4);
    const double2 *dw = reinterpret_cast<const double2 *>(dWa + (size_t)smap[b * P.g.nint + l] * 24);
    const double r4[4] = {rr.x, rr.y, rr.z, rr.w};
    double d4[4], ds = 0.0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {  // P_k(t) = sum_q dW[k][q] t^q and P_k'(t): 5 + 4 FMA
      const double2 c01 = __ldg(dw + 3 * k), c23 = __ldg(dw + 3 * k + 1), c45 = __ldg(dw + 3 * k + 2);
      double p = fma(c45.y, t, c45.x), dp = c45.y;
      dp = fma(dp, t, p);
      p = fma(p, t, c23.y);
      dp = fma(dp, t, p);
      p = fma(p, t, c23.x);
      dp = fma(dp, t, p);
      p = fma(p, t, c01.y);
      dp = fma(dp, t, p);
      d4[k] = fma(p, t, c01.x);
      ds = fma(r4[k], dp, ds);
    }
    dsrow[row] = clamped ? 0.0 : ds;
    st4(drow + (size_t)row * 4, d4[0], d4[1], d4[2], d4[3]);
  }
  // padded rows of each segment
  int off = 0;
  for (int b = 0; b < P.ntypes; ++b) {  // uniform
    for (int j = nvb[b] + lane; j < P.sel[b]; j += 32) {
      dsrow[off + j] = 0.0;
      st4(drow + (size_t)(off + j) * 4, 0.0, 0.0, 0.0, 0.0);
    }
    off += P.sel[b];
  }
}

// rows_kernel fused with the environment and the force back end (dp_tabulate_fusion_env_grad_tc_f64): a
// lane per valid row forms the row from coordinates (env_vals, as dp_env_mat), its dE/ds and dE/dR~ as
// rows_kernel does, and from them, in registers, the row's force contribution g = dE/d(x_j - x_i) by
// dp_force_virial's arithmetic: F_i += g, F_j -= g (atomics), virial -= d (x) g; s, R~, ds and dR~ never
// reach memory.  The per-atom sums are reduced over the warp and added once.
__global__ void __launch_bounds__(32 * kRowsWarps) rows_force_kernel(const RowsParams P) {
  __shared__ int nvbw[kRowsWarps][DP_MAX_TYPES];
  extern __shared__ short smapw[];  // [kRowsWarps][nkeys]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t a = (int64_t)blockIdx.x * kRowsWarps + warp;
  if (a >= P.natoms) return;  // warp-uniform
  int *nvb = nvbw[warp];
  short *smap = smapw + (size_t)warp * P.nkeys;
  const int64_t i = P.atom0 + a;
  const short *keys = P.keys + i * P.cap;
  const int nslot = P.nslots[i];
  for (int k = lane; k < P.nkeys; k += 32) smap[k] = -1;
  __syncwarp();
  for (int x = lane; x < nslot; x += 32) smap[keys[x]] = (short)x;  // the map of the atom's keys
  const int nv = env_valid_rows(P.env, P.nnei, P.sel, P.ntypes, i, lane, nvb, nullptr);  // (orders the map)
  const double *dWa = P.dW + (size_t)a * P.cap * 24;
  double f[3] = {0.0, 0.0, 0.0}, w[9];
#pragma unroll
  for (int x = 0; x < 9; ++x) w[x] = 0.0;
  for (int v = lane; v < nv; v += 32) {
    int b;
    const int row = valid_row(v, nvb, P.sel, P.ntypes, b);
    const int j = __ldg(P.env.nlist + i * P.nnei + row);
    const EnvVals ev = env_vals(P.env, i, j);
    double t;
    bool clamped;
    const int l = locate_fast(P.g, P.gf, P.nodes, ev.r4[0], t, clamped);
    const double2 *dw = reinterpret_cast<const double2 *>(dWa + (size_t)smap[b * P.g.nint + l] * 24);
    double d4[4], ds = 0.0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {  // as rows_kernel
      const double2 c01 = __ldg(dw + 3 * k), c23 = __ldg(dw + 3 * k + 1), c45 = __ldg(dw + 3 * k + 2);
      double p = fma(c45.y, t, c45.x), dp = c45.y;
      dp = fma(dp, t, p);
      p = fma(p, t, c23.y);
      dp = fma(dp, t, p);
      p = fma(p, t, c23.x);
      dp = fma(dp, t, p);
      p = fma(p, t, c01.y);
      dp = fma(dp, t, p);
      d4[k] = fma(p, t, c01.x);
      ds = fma(ev.r4[k], dp, ds);
    }
    ds = clamped ? 0.0 : ds;
    // as dp_force_virial: the s column feeds both the table input and R~[0]
    const double g0 = ds + d4[0];
    const double p = fma(d4[1], ev.d[0], fma(d4[2], ev.d[1], d4[3] * ev.d[2]));
    const double cd = fma(g0 * ev.dsv, ev.inv_r * P.env.inv_std,
                          (ev.dsv - ev.sv * ev.inv_r) * ev.inv_r * ev.inv_r * p * P.env.inv_std_all);
    const double ce = ev.sv * ev.inv_r * P.env.inv_std_all;
    const double g[3] = {fma(cd, ev.d[0], ce * d4[1]), fma(cd, ev.d[1], ce * d4[2]), fma(cd, ev.d[2], ce * d4[3])};
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      f[c] += g[c];
      atomicAdd(P.F + 3 * (int64_t)j + c, -g[c]);
    }
#pragma unroll
    for (int x = 0; x < 3; ++x)
#pragma unroll
      for (int y = 0; y < 3; ++y) w[3 * x + y] = fma(-ev.d[x], g[y], w[3 * x + y]);
  }
#pragma unroll
  for (int c = 0; c < 3; ++c)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) f[c] += __shfl_xor_sync(0xffffffffu, f[c], o);
#pragma unroll
  for (int x = 0; x < 9; ++x)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w[x] += __shfl_xor_sync(0xffffffffu, w[x], o);
  if (lane < 3) atomicAdd(P.F + 3 * i + lane, lane == 0 ? f[0] : lane == 1 ? f[1] : f[2]);
  if (lane < 9) {
    double vv = w[0];
#pragma unroll
    for (int x = 1; x < 9; ++x)
      if (lane == x) vv = w[x];
    atomicAdd(P.virial + lane, vv);
  }
}

int check_work(const Layout &L, const void *work, size_t nbytes, const char *who) {
  if (!work) return set_error(DP_ERR_NULL, "%s: work is NULL", who);
  if (nbytes < L.total) return set_error(DP_ERR_SHAPE, "%s: work holds %zu bytes, needs %zu", who, nbytes, L.total);
  if (reinterpret_cast<uintptr_t>(work) % 256) return set_error(DP_ERR_SHAPE, "%s: work is not 256-byte aligned", who);
  return DP_OK;
}

// Sizes of a plan for this geometry; DP_OK or an error (message set).
int plan_shape(const dp_table_info *info, int nnei, int ntypes, int M1, TableGeom *g, Shape *S, const char *who) {
  int rc = make_geom(info, g);
  if (rc) return rc;
  if (nnei < 1 || ntypes < 1 || ntypes > DP_MAX_TYPES || M1 < 1 || M1 > DP_MAX_M1)
    return set_error(DP_ERR_SHAPE, "%s: nnei %d, ntypes %d, M1 %d out of range", who, nnei, ntypes, M1);
  if ((int64_t)ntypes * g->nint > kMaxKeys)
    return set_error(DP_ERR_UNSUPPORTED, "%s: ntypes x nint = %lld intervals per centre type, at most %d", who,
                     (long long)ntypes * g->nint, kMaxKeys);
  *S = table_shape(*g, ntypes, M1);
  return DP_OK;
}

// The plan of a call: present, large enough and made for the call's geometry (checked on the host).
int check_plan(const dp_tc_plan *plan, const dp_table_info *info, int nnei, int ntypes, int M1, const Shape &S,
               const char *who) {
  if (!plan || !plan->data) return set_error(DP_ERR_NULL, "%s: plan is NULL", who);
  const dp_table_info &a = plan->info;
  if (a.lower != info->lower || a.upper != info->upper || a.upper_ext != info->upper_ext ||
      a.stride0 != info->stride0 || a.stride1 != info->stride1 || plan->nnei != nnei || plan->ntypes != ntypes ||
      plan->M1 != M1)
    return set_error(DP_ERR_SHAPE, "%s: the plan was made for another table info, nnei, ntypes or M1", who);
  if (plan->bytes < plan_layout(S).total) return set_error(DP_ERR_SHAPE, "%s: plan buffer too short", who);
  return DP_OK;
}

// C' of every centre type from the table, then its digit planes: forward A = C'^T (rows: the
// channels, K: 6 key + q), backward A = C' (rows: 6 key + q, K: the channels).
int make_plan(const double *table, const dp_table_info *info, int nnei, int ntypes, int M1, void *buf,
              size_t bytes, dp_tc_plan *out, void *stream) {
  clear_error();
  static const char *who = "dp_tabulate_tc_plan_f64";
  TableGeom g;
  Shape s{};
  int rc = plan_shape(info, nnei, ntypes, M1, &g, &s, who);
  if (rc) return rc;
  if (!table || !buf || !out) return set_error(DP_ERR_NULL, "%s: table, plan buffer or plan is NULL", who);
  const PlanLayout P = plan_layout(s);
  if (bytes < P.total) return set_error(DP_ERR_SHAPE, "%s: plan buffer holds %zu bytes, needs %zu", who, bytes, P.total);
  if (reinterpret_cast<uintptr_t>(buf) % 256) return set_error(DP_ERR_SHAPE, "%s: plan buffer is not 256-byte aligned", who);
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(buf);
  nodes_kernel<<<(unsigned)((g.nint + 256) / 256), 256, 0, st>>>(g, reinterpret_cast<double *>(wk + P.nodes));
  if ((rc = launch_status(who))) return rc;
  double *Cp = reinterpret_cast<double *>(wk + P.cp);
  const int64_t total = (int64_t)s.ntypes * s.Kp * s.M1;
  const unsigned cblocks = (unsigned)std::min<int64_t>((total + 255) / 256, 1 << 16);
  // forward: the u^q coefficients (the moments are in u, all K entries of a column of one scale)
  coef_kernel<<<cblocks, 256, 0, st>>>(table, g, s.ntypes, s.M1, s.Kp, 1.0 / (double)nnei, true, Cp);
  rc = launch_status(who);
  for (int t = 0; t < s.ntypes && !rc; ++t) {
    const double *Ct = Cp + (size_t)t * s.Kp * s.M1;
    rc = split_rows(Ct, 1, s.M1, s.M1, s.Kp, s.Mpf, s.Kp, kTM, wk + P.afwd + (size_t)t * kS * s.Mpf * s.Kp * 2,
                    wk + P.efwd + (size_t)t * s.Mpf * sizeof(int), st, who);
  }
  // backward: the t^q coefficients (each row 6 key + q of A has its own exponent), so that the rows
  // kernel evaluates its polynomials in t itself, with no 1/Delta on the way in or out
  if (!rc) {
    coef_kernel<<<cblocks, 256, 0, st>>>(table, g, s.ntypes, s.M1, s.Kp, 1.0 / (double)nnei, false, Cp);
    rc = launch_status(who);
  }
  for (int t = 0; t < s.ntypes && !rc; ++t) {
    const double *Ct = Cp + (size_t)t * s.Kp * s.M1;
    unsigned char *eb = wk + P.ebwd + (size_t)t * s.Mpb * sizeof(int);
    if (!rc && s.b8)
      rc = split_rows<Digits7x8>(Ct, s.M1, 1, s.Kp, s.M1, s.Mpb, s.Kpm, kTM,
                                 wk + P.abwd + (size_t)t * tb::kSB * s.Mpb * s.Kpm * 2, eb, st, who);
    else if (!rc)
      rc = split_rows(Ct, s.M1, 1, s.Kp, s.M1, s.Mpb, s.Kpm, kTM, wk + P.abwd + (size_t)t * kS * s.Mpb * s.Kpm * 2, eb,
                      st, who);
  }
  if (rc) return rc;
  out->data = buf;
  out->bytes = bytes;
  out->info = *info;
  out->nnei = nnei;
  out->ntypes = ntypes;
  out->M1 = M1;
  return DP_OK;
}

RunsParams runs_params(const double *s, const double *Rt, const int32_t *nvalid, const int32_t *atype,
                       const TableGeom &g, const Segments &seg, const Shape &S, const Layout &L, unsigned char *wk,
                       int nnei, const double *nodes) {
  RunsParams R{};
  R.s = s;
  R.Rt = Rt;
  R.nvalid = nvalid;
  R.atype = atype;
  R.g = g;
  R.gf = to_f32(g);
  R.nnei = nnei;
  R.ntypes = S.ntypes;
  R.nkeys = S.nkeys;
  R.cap = S.cap;
  R.nsl = S.nsl;
  R.tiles_all = S.tiles_all;
  for (int b = 0; b < DP_MAX_TYPES; ++b) R.sel[b] = seg.sel[b];
  R.keys = reinterpret_cast<short *>(wk + L.keys);
  R.nslots = reinterpret_cast<int *>(wk + L.nslots);
  R.occ = wk + L.occ;
  R.map = reinterpret_cast<int *>(wk + L.map);
  R.fexp = reinterpret_cast<int *>(wk + L.fexp);
  R.nodes = nodes;
  return R;
}

// Validation shared by the forward and the backward; fills g, seg, S, L.
int tc_args(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt, int64_t nloc,
            int nnei, int ntypes, const int32_t *sel, int M1, const void *out0, const void *out1, void *work,
            size_t work_bytes, TableGeom *g, Segments *seg, Shape *S, Layout *L, const char *who) {
  int rc = check_fusion_args(plan ? plan->data : nullptr, info, s, Rt, nloc, nnei, ntypes, sel, M1, out0, out1, g, seg);
  if (rc || nloc == 0) return rc;
  Shape T{};
  if ((rc = plan_shape(info, nnei, ntypes, M1, g, &T, who))) return rc;
  if ((rc = check_plan(plan, info, nnei, ntypes, M1, T, who))) return rc;
  *S = make_shape(*g, nloc, nnei, ntypes, M1);
  *L = make_layout(*S);
  if ((rc = check_work(*L, work, work_bytes, who))) return rc;
  return tg::set_smem(who);
}

// env: the rows come from coordinates (dp_tabulate_fusion_env_fwd_tc_f64; s, Rt and nvalid unused, the
// counts of valid rows written to nvalid_out when given).
int fwd(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt, const int32_t *nvalid,
        const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1, double *T, int M2,
        double *D, void *work, size_t work_bytes, void *stream, const EnvRow *env = nullptr,
        int32_t *nvalid_out = nullptr, const char *who = "dp_tabulate_fusion_fwd_tc_f64") {
  clear_error();
  TableGeom g;
  Segments seg;
  Shape S{};
  Layout L{};
  if (D && (M2 < 1 || M2 > M1)) return set_error(DP_ERR_SHAPE, "%s: M2 %d not in 1 .. M1 = %d", who, M2, M1);
  int rc = tc_args(plan, info, s, Rt, nloc, nnei, ntypes, sel, M1, T, T, work, work_bytes, &g, &seg, &S, &L, who);
  if (rc || nloc == 0) return rc;
  const PlanLayout PL = plan_layout(S);
  const unsigned char *pk = static_cast<const unsigned char *>(plan->data);
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(work);
  prof_mark("tc_fwd", st);
  if (cudaMemsetAsync(wk + L.occ, 0, (size_t)ntypes * S.tiles_all * S.nsl, st) != cudaSuccess)
    return set_error(DP_ERR_CUDA, "%s: cudaMemsetAsync: %s", who, cudaGetErrorString(cudaGetLastError()));
  RunsParams R = runs_params(s, Rt, nvalid, atype, g, seg, S, L, wk, nnei,
                             reinterpret_cast<const double *>(pk + PL.nodes));
  R.W = reinterpret_cast<double *>(wk + L.w);
  if (env) {
    R.env = *env;
    R.nvalid_out = nvalid_out;
  }
  longlong2 *part = reinterpret_cast<longlong2 *>(wk + L.part);
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(cudaGetLastError()));
  const int ncta = std::max(1, std::min(nsm, kMaxCtasF));
  for (int64_t c0 = 0; c0 < nloc; c0 += S.chunk) {
    const int64_t n = std::min<int64_t>(S.chunk, nloc - c0);
    const int64_t Np = round_up(kCols * n, kTN), ntiles = Np / kTN, tile0 = c0 / kTileAtoms;
    R.atom0 = c0;
    R.natoms = n;
    const dim3 rgrid((unsigned)((n + kRunsWarps - 1) / kRunsWarps));
    if (env)
      runs_kernel<true, true><<<rgrid, 32 * kRunsWarps, kRunsWarps * S.nkeys * sizeof(short), st>>>(R);
    else
      runs_kernel<true><<<rgrid, 32 * kRunsWarps, kRunsWarps * S.nkeys * sizeof(short), st>>>(R);
    if ((rc = launch_status(who))) return rc;
    prof_mark("tc_runs_moments", st);
    const int64_t nlist = (int64_t)ntypes * ntiles;
    slice_list_kernel<<<(unsigned)((nlist + 3) / 4), 128, 0, st>>>(wk + L.occ, S.tiles_all, tile0, ntiles, ntypes,
                                                                    S.nsl, reinterpret_cast<short *>(wk + L.slist),
                                                                    reinterpret_cast<int *>(wk + L.scount));
    if ((rc = launch_status(who))) return rc;
    const int nmt = S.Mpf / kTM;
    fwd_schedule_kernel<<<1, 1024, 0, st>>>(reinterpret_cast<const int *>(wk + L.scount), nlist * nmt, ntiles, nmt, ncta,
                                            reinterpret_cast<int4 *>(wk + L.pieces), reinterpret_cast<int *>(wk + L.pcta),
                                            reinterpret_cast<int *>(wk + L.cta_start),
                                            reinterpret_cast<int *>(wk + L.npieces),
                                            reinterpret_cast<int *>(wk + L.pfirst));
    if ((rc = launch_status(who))) return rc;
    prof_mark("tc_slice_lists", st);
    tg::Params G{};
    G.fwd = true;
    G.aplanes = pk + PL.afwd;
    G.astride = (size_t)kS * S.Mpf * S.Kp * 2;
    G.Eexp = reinterpret_cast<const int *>(pk + PL.efwd);
    G.estride = S.Mpf;
    G.ka = S.nsl;
    G.nmt = nmt;
    G.W = R.W;  // B made from the moments inside the GEMM
    G.map = R.map;
    G.nkeys = S.nkeys;
    G.cap = S.cap;
    G.Fexp = R.fexp;
    G.ntiles = ntiles;
    G.Np = Np;
    G.Mp = S.Mpf;
    G.slist = reinterpret_cast<const short *>(wk + L.slist);
    G.scount = reinterpret_cast<const int *>(wk + L.scount);
    G.zmax = S.zmax;
    G.part = part;
    G.tout = T;  // items in one piece write T themselves
    G.pieces = reinterpret_cast<const int4 *>(wk + L.pieces);
    G.cta_start = reinterpret_cast<const int *>(wk + L.cta_start);
    G.ldt = M1;
    G.atype = atype;
    G.natoms = n;
    G.atom0 = c0;
    G.ntypes = ntypes;
    if ((rc = tg::launch(G, st, who, ncta))) return rc;
    prof_mark("tc_gemm_fwd", st);
    fwd_finish_kernel<<<(unsigned)n, 128, D ? (size_t)kCols * M1 * sizeof(double) : 0, st>>>(
        part, S.Mpf, G.Eexp, R.fexp, reinterpret_cast<const int *>(wk + L.npieces),
        reinterpret_cast<const int *>(wk + L.pfirst), ntiles, nmt, c0, atype, ntypes, M1, T, M2, D);
    if ((rc = launch_status(who))) return rc;
    prof_mark("tc_finish_fwd", st);
  }
  return DP_OK;
}

// env: the rows come from coordinates and the rows kernel adds the forces and virial instead of writing
// ds and dRt (dp_tabulate_fusion_env_grad_tc_f64; s, Rt, nvalid, ds and dRt unused; F [nall][3] and
// virial [9] are zeroed first).
int grad(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt, const int32_t *nvalid,
         const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1, const double *dT,
         double *ds, double *dRt, void *work, size_t work_bytes, int flags, void *stream, const EnvRow *env = nullptr,
         double *F = nullptr, double *virial = nullptr, int64_t nall = 0,
         const char *who = "dp_tabulate_fusion_grad_tc_f64") {
  clear_error();
  if (flags & ~DP_TC_REUSE_RUNS) return set_error(DP_ERR_SHAPE, "%s: unknown flags %#x", who, flags);
  TableGeom g;
  Segments seg;
  Shape S{};
  Layout L{};
  int rc = tc_args(plan, info, s, Rt, nloc, nnei, ntypes, sel, M1, env ? (void *)F : ds, env ? (void *)virial : dRt,
                   work, work_bytes, &g, &seg, &S, &L, who);
  if (rc) return rc;
  if (env) {  // the forces and virial are sums: zeroed first, also for nloc = 0
    cudaError_t e = cudaMemsetAsync(virial, 0, 9 * sizeof(double), (cudaStream_t)stream);
    if (e == cudaSuccess && nall > 0) e = cudaMemsetAsync(F, 0, (size_t)nall * 3 * sizeof(double), (cudaStream_t)stream);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
  }
  if (nloc == 0) return DP_OK;
  if (!dT) return set_error(DP_ERR_NULL, "%s: dT is NULL", who);
  const PlanLayout PL = plan_layout(S);
  const unsigned char *pk = static_cast<const unsigned char *>(plan->data);
  const cudaStream_t st = (cudaStream_t)stream;
  unsigned char *wk = static_cast<unsigned char *>(work);
  const bool reuse = (flags & DP_TC_REUSE_RUNS) != 0;
  prof_mark("tc_grad", st);
  if (!reuse && cudaMemsetAsync(wk + L.occ, 0, (size_t)ntypes * S.tiles_all * S.nsl, st) != cudaSuccess)
    return set_error(DP_ERR_CUDA, "%s: cudaMemsetAsync: %s", who, cudaGetErrorString(cudaGetLastError()));
  RunsParams R = runs_params(s, Rt, nvalid, atype, g, seg, S, L, wk, nnei,
                             reinterpret_cast<const double *>(pk + PL.nodes));
  const int mtiles = S.Mpb / kTM;
  double *dW = reinterpret_cast<double *>(wk + L.w);
  RowsParams Q{};
  Q.s = s;
  Q.Rt = Rt;
  Q.nvalid = nvalid;
  Q.atype = atype;
  Q.g = g;
  Q.gf = R.gf;
  Q.nodes = R.nodes;
  Q.nnei = nnei;
  Q.ntypes = ntypes;
  Q.nkeys = S.nkeys;
  Q.cap = S.cap;
  for (int b = 0; b < DP_MAX_TYPES; ++b) Q.sel[b] = seg.sel[b];
  Q.keys = R.keys;
  Q.nslots = R.nslots;
  Q.dW = dW;
  Q.ds = ds;
  Q.dRt = dRt;
  if (env) {
    R.env = *env;
    Q.env = *env;
    Q.F = F;
    Q.virial = virial;
  }
  for (int64_t c0 = 0; c0 < nloc; c0 += S.chunk) {
    const int64_t n = std::min<int64_t>(S.chunk, nloc - c0);
    const int64_t Np = round_up(kCols * n, kTN), ntiles = Np / kTN, tile0 = c0 / kTileAtoms;
    R.atom0 = c0;
    R.natoms = n;
    if (!reuse) {
      const dim3 rgrid((unsigned)((n + kRunsWarps - 1) / kRunsWarps));
      if (env)
        runs_kernel<false, true><<<rgrid, 32 * kRunsWarps, kRunsWarps * S.nkeys * sizeof(short), st>>>(R);
      else
        runs_kernel<false><<<rgrid, 32 * kRunsWarps, kRunsWarps * S.nkeys * sizeof(short), st>>>(R);
      if ((rc = launch_status(who))) return rc;
      prof_mark("tc_runs", st);
    }
    if (S.b8) {
      // B = dT^T on 8-atom tiles in the 7 x 8-bit digits: the columns 4 a + k are the rows of this chunk's dT
      if ((rc = split_rows_1k<Digits7x8>(dT + c0 * kCols * M1, M1, 1, kCols * n, M1, round_up(kCols * n, tb::kTNB),
                                         S.Kpm, tb::kTNB, wk + L.bplanes, wk + L.fexp, st, who)))
        return rc;
      prof_mark("tc_split_dT", st);
      if (cudaMemsetAsync(wk + L.nunits, 0, (size_t)ntypes * sizeof(int), st) != cudaSuccess)
        return set_error(DP_ERR_CUDA, "%s: cudaMemsetAsync: %s", who, cudaGetErrorString(cudaGetLastError()));
      const int64_t ntiles8 = (n + tb::kAtomsB - 1) / tb::kAtomsB, nlist = (int64_t)ntypes * ntiles8;
      bwd_units8_kernel<<<(unsigned)nlist, 32 * tb::kAtomsB, 0, st>>>(
          R.keys, R.nslots, atype, ntypes, S.cap, c0, n, ntiles8, S.maxunits8, reinterpret_cast<int *>(wk + L.units),
          reinterpret_cast<int *>(wk + L.nunits));
      if ((rc = launch_status(who))) return rc;
      prof_mark("tc_units", st);
      for (int t = 0; t < ntypes; ++t) {
        tb::Params G{};
        G.aplanes = pk + PL.abwd + (size_t)t * tb::kSB * S.Mpb * S.Kpm * 2;
        G.Eexp = reinterpret_cast<const int *>(pk + PL.ebwd) + (size_t)t * S.Mpb;
        G.ka = S.Kpm / kTK;
        G.bplanes = wk + L.bplanes;
        G.Fexp = R.fexp;
        G.Mp = S.Mpb;
        G.scat = dW;
        G.keys = R.keys;
        G.nslots = R.nslots;
        G.cap = S.cap;
        G.nkeys = S.nkeys;
        G.kq = kQ;
        G.atype = atype;
        G.natoms = n;
        G.atom0 = c0;
        G.alpha = t;
        G.ntypes = ntypes;
        G.units = reinterpret_cast<const int *>(wk + L.units) + (size_t)t * S.maxunits8;
        G.nunits = reinterpret_cast<const int *>(wk + L.nunits) + t;
        if ((rc = tb::launch(G, st, who))) return rc;
        prof_mark("tc_gemm_grad", st);
      }
    } else {
      // B = dT^T: the columns 4 a + k are the rows of this chunk's dT
      if ((rc = split_rows(dT + c0 * kCols * M1, M1, 1, kCols * n, M1, Np, S.Kpm, kTN, wk + L.bplanes, wk + L.fexp, st,
                           who)))
        return rc;
      prof_mark("tc_split_dT", st);
      if (cudaMemsetAsync(wk + L.nunits, 0, (size_t)ntypes * sizeof(int), st) != cudaSuccess)
        return set_error(DP_ERR_CUDA, "%s: cudaMemsetAsync: %s", who, cudaGetErrorString(cudaGetLastError()));
      const int64_t nlist = (int64_t)ntypes * ntiles;
      bwd_units_kernel<<<(unsigned)((nlist + 127) / 128), 128, 0, st>>>(wk + L.occ, S.tiles_all, tile0, ntiles, ntypes,
                                                                        S.nsl, mtiles, S.maxunits,
                                                                        reinterpret_cast<int *>(wk + L.units),
                                                                        reinterpret_cast<int *>(wk + L.nunits));
      if ((rc = launch_status(who))) return rc;
      prof_mark("tc_units", st);
      for (int t = 0; t < ntypes; ++t) {
        tg::Params G{};
        G.fwd = false;
        G.aplanes = pk + PL.abwd + (size_t)t * kS * S.Mpb * S.Kpm * 2;
        G.Eexp = reinterpret_cast<const int *>(pk + PL.ebwd) + (size_t)t * S.Mpb;
        G.ka = S.Kpm / kTK;
        G.nmt = mtiles;
        G.bplanes = wk + L.bplanes;
        G.Fexp = R.fexp;
        G.ntiles = ntiles;
        G.Np = Np;
        G.Mp = S.Mpb;
        G.sflags = wk + L.occ + ((size_t)t * S.tiles_all + tile0) * S.nsl;
        G.nsf = S.nsl;
        G.scat = dW;
        G.keys = R.keys;
        G.nslots = R.nslots;
        G.cap = S.cap;
        G.nkeys = S.nkeys;
        G.kq = kQ;
        G.atype = atype;
        G.natoms = n;
        G.atom0 = c0;
        G.alpha = t;
        G.ntypes = ntypes;
        G.units = reinterpret_cast<const int *>(wk + L.units) + (size_t)t * S.maxunits;
        G.nunits = reinterpret_cast<const int *>(wk + L.nunits) + t;
        if ((rc = tg::launch(G, st, who))) return rc;
        prof_mark("tc_gemm_grad", st);
      }
    }
    Q.atom0 = c0;
    Q.natoms = n;
    const dim3 qgrid((unsigned)((n + kRowsWarps - 1) / kRowsWarps));
    if (env)
      rows_force_kernel<<<qgrid, 32 * kRowsWarps, kRowsWarps * S.nkeys * sizeof(short), st>>>(Q);
    else
      rows_kernel<<<qgrid, 32 * kRowsWarps, kRowsWarps * S.nkeys * sizeof(short), st>>>(Q);
    if ((rc = launch_status(who))) return rc;
    prof_mark("tc_rows", st);
  }
  return DP_OK;
}

EnvRow env_row(const dp_env_info *e, const double *coord, const int32_t *nlist) {
  EnvRow E{};
  E.coord = coord;
  E.nlist = nlist;
  E.rcs = e->rcs;
  E.rc = e->rc;
  E.inv_width = 1.0 / (e->rc - e->rcs);
  E.mean = e->mean;
  E.inv_std = 1.0 / e->std;
  E.inv_std_all = 1.0 / e->std_all;
  E.kind = e->kind;
  return E;
}

int env_fwd(const dp_tc_plan *plan, const dp_table_info *info, const double *coord, const int32_t *nlist,
            const dp_env_info *env, const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel,
            int M1, int32_t *nvalid, double *T, int M2, double *D, void *work, size_t work_bytes, void *stream) {
  clear_error();
  static const char *who = "dp_tabulate_fusion_env_fwd_tc_f64";
  if (int rc = check_env(env)) return rc;
  const EnvRow E = env_row(env, coord, nlist);
  // coord and nlist stand where the plain call's s and Rt are checked for NULL
  return fwd(plan, info, coord, reinterpret_cast<const double *>(nlist), nullptr, atype, nloc, nnei, ntypes, sel, M1,
             T, M2, D, work, work_bytes, stream, &E, nvalid, who);
}

int env_grad(const dp_tc_plan *plan, const dp_table_info *info, const double *coord, const int32_t *nlist,
             const dp_env_info *env, const int32_t *atype, int64_t nloc, int64_t nall, int nnei, int ntypes,
             const int32_t *sel, int M1, const double *dT, double *F, double *virial, void *work, size_t work_bytes,
             int flags, void *stream) {
  clear_error();
  static const char *who = "dp_tabulate_fusion_env_grad_tc_f64";
  if (int rc = check_env(env)) return rc;
  if (nall < nloc) return set_error(DP_ERR_SHAPE, "%s: nall = %lld < nloc = %lld", who, (long long)nall, (long long)nloc);
  if (!virial || (nall > 0 && !F)) return set_error(DP_ERR_NULL, "%s: NULL output", who);
  const EnvRow E = env_row(env, coord, nlist);
  return grad(plan, info, coord, reinterpret_cast<const double *>(nlist), nullptr, atype, nloc, nnei, ntypes, sel, M1,
              dT, nullptr, nullptr, work, work_bytes, flags, stream, &E, F, virial, nall, who);
}

size_t work_bytes_api(const dp_table_info *info, int64_t nloc, int nnei, int ntypes, int M1) {
  clear_error();
  TableGeom g;
  Shape S{};
  if (nloc < 0) {
    set_error(DP_ERR_SHAPE, "dp_tabulate_tc_work_bytes: nloc %lld < 0", (long long)nloc);
    return 0;
  }
  if (plan_shape(info, nnei, ntypes, M1, &g, &S, "dp_tabulate_tc_work_bytes")) return 0;
  return make_layout(make_shape(g, nloc, nnei, ntypes, M1)).total;
}

size_t plan_bytes_api(const dp_table_info *info, int nnei, int ntypes, int M1) {
  clear_error();
  TableGeom g;
  Shape S{};
  if (plan_shape(info, nnei, ntypes, M1, &g, &S, "dp_tabulate_tc_plan_bytes")) return 0;
  return plan_layout(S).total;
}

}  // namespace tt
}  // namespace

// This unit's GEMM wait timeouts (see tc_gemm.cuh), for dp_tc_wait_timeouts.
int take_wait_timeouts_tabulate(unsigned int *count) { return tc::take_wait_timeouts(count); }

}  // namespace dpc

extern "C" {

size_t dp_tabulate_tc_work_bytes(const dp_table_info *info, int64_t nloc, int nnei, int ntypes, int M1) {
  return dpc::tt::work_bytes_api(info, nloc, nnei, ntypes, M1);
}

size_t dp_tabulate_tc_plan_bytes(const dp_table_info *info, int nnei, int ntypes, int M1) {
  return dpc::tt::plan_bytes_api(info, nnei, ntypes, M1);
}

int dp_tabulate_tc_plan_f64(const double *table, const dp_table_info *info, int nnei, int ntypes, int M1, void *buf,
                            size_t bytes, dp_tc_plan *plan, void *stream) {
  return dpc::tt::make_plan(table, info, nnei, ntypes, M1, buf, bytes, plan, stream);
}

int dp_tabulate_fusion_fwd_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt,
                                  const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                  const int32_t *sel, int M1, double *T, int M2, double *D, void *work,
                                  size_t work_bytes, void *stream) {
  return dpc::tt::fwd(plan, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, T, M2, D, work, work_bytes,
                      stream);
}

int dp_tabulate_fusion_env_fwd_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *coord,
                                      const int32_t *nlist, const dp_env_info *env, const int32_t *atype, int64_t nloc,
                                      int nnei, int ntypes, const int32_t *sel, int M1, int32_t *nvalid, double *T,
                                      int M2, double *D, void *work, size_t work_bytes, void *stream) {
  return dpc::tt::env_fwd(plan, info, coord, nlist, env, atype, nloc, nnei, ntypes, sel, M1, nvalid, T, M2, D, work,
                          work_bytes, stream);
}

int dp_tabulate_fusion_env_grad_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *coord,
                                       const int32_t *nlist, const dp_env_info *env, const int32_t *atype,
                                       int64_t nloc, int64_t nall, int nnei, int ntypes, const int32_t *sel, int M1,
                                       const double *dT, double *F, double *virial, void *work, size_t work_bytes,
                                       int flags, void *stream) {
  return dpc::tt::env_grad(plan, info, coord, nlist, env, atype, nloc, nall, nnei, ntypes, sel, M1, dT, F, virial,
                           work, work_bytes, flags, stream);
}

int dp_tabulate_fusion_grad_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt,
                                   const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                   const int32_t *sel, int M1, const double *dT, double *ds, double *dRt, void *work,
                                   size_t work_bytes, int flags, void *stream) {
  return dpc::tt::grad(plan, info, s, Rt, nvalid, atype, nloc, nnei, ntypes, sel, M1, dT, ds, dRt, work, work_bytes,
                       flags, stream);
}

}  // extern "C"
