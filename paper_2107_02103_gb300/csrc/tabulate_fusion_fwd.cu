// Fused tabulated embedding + contraction, forward (Sec. II, kernel fusion):
//   T_i[k][m] = (1/N_c) sum over valid rows j of R~_ij[k] * g_m(s_ij)
// G_i is never stored: each row's M1 polynomial values live in registers
// only for the four FMAs that fold them into T_i.  Padded rows are skipped
// through the per-type valid counts.
//
// GB300 design.  The FP64 pipe issues one warp instruction per 16 SM clocks
// no matter how many lanes are active, so the mapping is chosen to keep every
// lane of every FP64 instruction busy:
//   * one warp per atom; the warp's 32 lanes are G = 32/CL groups of CL
//     channel lanes; group g takes every G-th valid neighbour, lane c of the
//     group owns channels c, c + CL, ..., c + (R-1) CL (R rounds).  For M1 =
//     100, CL = 8 and R = 13 fill 104 slots for 100 channels (96 %), against
//     78 % for one neighbour per warp instruction.
//   * the interval search, the segment lookup and the R~ row load are done
//     once per neighbour, spread over the lanes (lane l handles neighbour
//     base + l) and handed to the groups through shared memory, so their
//     FP64 work costs 1/32 of an instruction per neighbour;
//   * the G partial T_i are summed with xor shuffles once per atom.
// Coefficients are read through the read-only path (the tables are a few MB
// and stay resident in the 126 MB L2).
#include <utility>

#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kFwdWarps = 4;

template <typename real>
struct FwdParams {
  const real *__restrict__ table;
  const real *__restrict__ s;
  const real *__restrict__ Rt;
  const int32_t *__restrict__ nvalid;
  const int32_t *__restrict__ atype;
  real *__restrict__ T;
  TableGeom geom;
  int64_t nloc;
  int32_t nnei, ntypes, M1, pair_stride;  // pair_stride = nint * M1 * 6
  int32_t sel[DP_MAX_TYPES];
  real inv_nnei;
};

template <typename real>
struct alignas(16) Stage {
  real r[32][4];    // R~ rows of the staged neighbours
  real t[32];       // local variable t
  int32_t off[32];  // element offset of the interval's coefficient row in the centre type's tables
};

template <typename real, int CL, int R>
__global__ void __launch_bounds__(kFwdWarps * 32) fwd_kernel(const FwdParams<real> P) {
  constexpr int G = 32 / CL;
  __shared__ Stage<real> stage[kFwdWarps];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t i = (int64_t)blockIdx.x * kFwdWarps + w;
  if (i >= P.nloc) return;  // warp-uniform
  Stage<real> &st = stage[w];
  const int g = lane / CL, c = lane % CL;

  // valid rows per type segment (clamped into [0, sel]) and their total
  int nvb[DP_MAX_TYPES];
  int nv = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q) {
    int x = 0;
    if (q < P.ntypes) x = clampi(P.nvalid ? __ldg(P.nvalid + i * P.ntypes + q) : P.sel[q], 0, P.sel[q]);
    nvb[q] = x;
    nv += x;
  }
  const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
  const real *__restrict__ tab = P.table + (size_t)alpha * P.ntypes * P.pair_stride;
  const real *__restrict__ srow = P.s + i * P.nnei;
  const real *__restrict__ Rrow = P.Rt + i * P.nnei * 4;

  real acc[R][4];
#pragma unroll
  for (int r = 0; r < R; ++r) acc[r][0] = acc[r][1] = acc[r][2] = acc[r][3] = real(0);

  for (int base = 0; base < nv; base += 32) {
    // stage: lane l prepares valid neighbour base + l
    const int v = base + lane;
    if (v < nv) {
      int b = 0, cum = 0, lim = nvb[0], off = 0;
#pragma unroll
      for (int q = 1; q < DP_MAX_TYPES; ++q)
        if (q < P.ntypes && v >= lim) {
          b = q;
          cum = lim;
          lim += nvb[q];
          off += P.sel[q - 1];
        }
      const int row = off + (v - cum);
      const Vec4<real> rr = ld4(Rrow + (size_t)row * 4);
      double t;
      bool clamped;
      const int l = locate(P.geom, (double)__ldg(srow + row), t, clamped);
      st.r[lane][0] = rr.x;
      st.r[lane][1] = rr.y;
      st.r[lane][2] = rr.z;
      st.r[lane][3] = rr.w;
      st.t[lane] = (real)t;
      st.off[lane] = (b * P.geom.nint + l) * P.M1 * 6;
    }
    __syncwarp();
    const int cnt = min(32, nv - base);
    for (int q = 0; q < cnt; q += G) {
      const int u = q + g;
      if (u < cnt) {
        const real t = st.t[u];
        const real r0 = st.r[u][0], r1 = st.r[u][1], r2 = st.r[u][2], r3 = st.r[u][3];
        const real *__restrict__ cp = tab + st.off[u] + c * 6;
#pragma unroll
        for (int r = 0; r < R; ++r) {
          if (r < R - 1 || c + r * CL < P.M1) {
            real cf[6];
            ld6(cp + r * CL * 6, cf);
            // g = ((((a t + b) t + c) t + d) t + e) t + f
            real gv = fma(cf[0], t, cf[1]);
            gv = fma(gv, t, cf[2]);
            gv = fma(gv, t, cf[3]);
            gv = fma(gv, t, cf[4]);
            gv = fma(gv, t, cf[5]);
            acc[r][0] = fma(r0, gv, acc[r][0]);
            acc[r][1] = fma(r1, gv, acc[r][1]);
            acc[r][2] = fma(r2, gv, acc[r][2]);
            acc[r][3] = fma(r3, gv, acc[r][3]);
          }
        }
      }
    }
    __syncwarp();
  }

  // sum the G groups' partial T_i
#pragma unroll
  for (int sh = CL; sh < 32; sh <<= 1)
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int k = 0; k < 4; ++k) acc[r][k] += __shfl_xor_sync(0xffffffffu, acc[r][k], sh);

  if (g == 0) {
    real *__restrict__ Ti = P.T + i * 4 * P.M1;
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int m = c + r * CL;
      if (m < P.M1)
#pragma unroll
        for (int k = 0; k < 4; ++k) Ti[k * P.M1 + m] = acc[r][k] * P.inv_nnei;
    }
  }
}

template <typename real>
using FwdKernel = void (*)(const FwdParams<real>);

template <typename real, int CL, int... Rs>
FwdKernel<real> pick_fwd(int R, std::integer_sequence<int, Rs...>) {
  FwdKernel<real> k = nullptr;
  ((R == Rs + 1 ? (k = &fwd_kernel<real, CL, Rs + 1>, 0) : 0), ...);
  return k;
}

// Channel-lane width CL and rounds R for M1: the pair with the fewest idle
// lane slots (CL = 8 costs a small group reduction, so it must win by >1 %).
void choose_fwd_shape(int M1, int *CL, int *R) {
  const int r32 = (M1 + 31) / 32, r8 = (M1 + 7) / 8;
  const double e32 = r32 <= 8 ? (double)M1 / (32.0 * r32) : -1.0;
  const double e8 = r8 <= 16 ? (double)M1 / (8.0 * r8) - 0.01 : -1.0;
  if (e8 > e32) {
    *CL = 8;
    *R = r8;
  } else {
    *CL = 32;
    *R = r32;
  }
}

template <typename real>
int fwd(const real *table, const dp_table_info *info, const real *s, const real *Rt, const int32_t *nvalid,
        const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1, real *T, void *stream) {
  clear_error();
  TableGeom g;
  Segments seg;
  int rc = check_fusion_args(table, info, s, Rt, nloc, nnei, ntypes, sel, M1, T, T, &g, &seg);
  if (rc) return rc;
  if (nloc == 0) return DP_OK;
  FwdParams<real> P;
  P.table = table;
  P.s = s;
  P.Rt = Rt;
  P.nvalid = nvalid;
  P.atype = atype;
  P.T = T;
  P.geom = g;
  P.nloc = nloc;
  P.nnei = nnei;
  P.ntypes = ntypes;
  P.M1 = M1;
  P.pair_stride = g.nint * M1 * 6;
  for (int b = 0; b < DP_MAX_TYPES; ++b) P.sel[b] = seg.sel[b];
  P.inv_nnei = (real)(1.0 / (double)nnei);
  int CL, R;
  choose_fwd_shape(M1, &CL, &R);
  FwdKernel<real> k = CL == 8 ? pick_fwd<real, 8>(R, std::make_integer_sequence<int, 16>{})
                              : pick_fwd<real, 32>(R, std::make_integer_sequence<int, 8>{});
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

}  // extern "C"
