// Backward of the fused forward: from dT_i = dE/dT_i,
//   dE/dR~_ij[k] = (1/N_c) sum_m dT_i[k][m] g_m(s_ij)
//   dE/ds_ij     = (1/N_c) sum_m (sum_k dT_i[k][m] R~_ij[k]) g'_m(s_ij)
// for valid rows, zero on padding rows (Sec. II: the compressed model serves
// the backward propagation that yields forces and virials).
//
// GB300 design.  Every output of this pass belongs to one neighbour row, so
// the lanes run over neighbours instead of channels: thread = one valid row,
// looping over the M1 channels.  Nothing is reduced across lanes -- a
// channel-parallel mapping would need five cross-lane sums per neighbour,
// each one a full-price FP64 warp instruction per shuffle level.  Per
// channel a thread evaluates g and g' together by Horner's rule (9 FMA),
// forms r_m = sum_k dT[k][m] R~[k] (4), and accumulates ds (1) and dR~ (4):
// 18 FP64 operations, all useful.  dT_i is staged once per block in shared
// memory as [M1][4] and read as broadcasts; each thread gathers its own
// interval's coefficient row, which walks contiguous memory as m advances.
// Valid rows of all type segments are packed into consecutive threads so
// only the last warp of an atom can idle; padding rows are zero-filled by
// the threads past the valid ones.
#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kGradThreads = 128;

template <typename real>
struct GradParams {
  const real *__restrict__ table;
  const real *__restrict__ s;
  const real *__restrict__ Rt;
  const int32_t *__restrict__ nvalid;
  const int32_t *__restrict__ atype;
  const real *__restrict__ dT;
  real *__restrict__ ds;
  real *__restrict__ dRt;
  TableGeom geom;
  int64_t nloc;
  int32_t nnei, ntypes, M1, pair_stride;
  int32_t sel[DP_MAX_TYPES];
  real inv_nnei;
};

template <typename real>
__global__ void __launch_bounds__(kGradThreads) grad_kernel(const GradParams<real> P) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  real *dTs = reinterpret_cast<real *>(smem_raw);  // [M1][4]
  const int64_t i = blockIdx.x;
  const int v = blockIdx.y * kGradThreads + threadIdx.x;  // packed row index of this thread

  int nvb[DP_MAX_TYPES];
  int nv = 0;
#pragma unroll
  for (int q = 0; q < DP_MAX_TYPES; ++q) {
    int x = 0;
    if (q < P.ntypes) x = clampi(P.nvalid ? __ldg(P.nvalid + i * P.ntypes + q) : P.sel[q], 0, P.sel[q]);
    nvb[q] = x;
    nv += x;
  }
  real *__restrict__ ds_i = P.ds + i * P.nnei;
  real *__restrict__ dR_i = P.dRt + i * P.nnei * 4;

  if ((int)(blockIdx.y * kGradThreads) < nv) {  // block-uniform
    const real *__restrict__ dTi = P.dT + i * 4 * P.M1;
    for (int e = threadIdx.x; e < 4 * P.M1; e += kGradThreads) {
      const int k = e / P.M1, m = e - k * P.M1;
      dTs[m * 4 + k] = __ldg(dTi + e);
    }
    __syncthreads();
  }

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
    const int alpha = P.atype ? clampi(__ldg(P.atype + i), 0, P.ntypes - 1) : 0;
    const Vec4<real> rr = ld4(P.Rt + (i * P.nnei + row) * 4);
    double td;
    bool clamped;
    const int l = locate(P.geom, (double)__ldg(P.s + i * P.nnei + row), td, clamped);
    const real t = (real)td;
    const real *__restrict__ cp =
        P.table + (size_t)(alpha * P.ntypes + b) * P.pair_stride + (size_t)l * P.M1 * 6;
    real a_ds = real(0), a0 = real(0), a1 = real(0), a2 = real(0), a3 = real(0);
#pragma unroll 2
    for (int m = 0; m < P.M1; ++m) {
      real cf[6];
      ld6(cp + m * 6, cf);
      const real d0 = dTs[m * 4 + 0], d1 = dTs[m * 4 + 1], d2 = dTs[m * 4 + 2], d3 = dTs[m * 4 + 3];
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
      a0 = fma(d0, p, a0);
      a1 = fma(d1, p, a1);
      a2 = fma(d2, p, a2);
      a3 = fma(d3, p, a3);
    }
    if (clamped) a_ds = real(0);
    ds_i[row] = a_ds * P.inv_nnei;
    st4(dR_i + (size_t)row * 4, a0 * P.inv_nnei, a1 * P.inv_nnei, a2 * P.inv_nnei, a3 * P.inv_nnei);
  } else if (v < P.nnei) {
    // padding row number v - nv, packed over the segments' padded tails
    const int w = v - nv;
    int b = 0, cum = 0, lim = P.sel[0] - nvb[0], off = 0;
#pragma unroll
    for (int q = 1; q < DP_MAX_TYPES; ++q)
      if (q < P.ntypes && w >= lim) {
        b = q;
        cum = lim;
        lim += P.sel[q] - nvb[q];
        off += P.sel[q - 1];
      }
    const int row = off + nvb[b] + (w - cum);
    ds_i[row] = real(0);
    st4(dR_i + (size_t)row * 4, real(0), real(0), real(0), real(0));
  }
}

template <typename real>
int grad(const real *table, const dp_table_info *info, const real *s, const real *Rt, const int32_t *nvalid,
         const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1, const real *dT,
         real *ds, real *dRt, void *stream) {
  clear_error();
  TableGeom g;
  Segments seg;
  int rc = check_fusion_args(table, info, s, Rt, nloc, nnei, ntypes, sel, M1, ds, dRt, &g, &seg);
  if (rc) return rc;
  if (nloc == 0) return DP_OK;
  if (!dT) return set_error(DP_ERR_NULL, "dT is NULL");
  if (nloc > 2147483647LL) return set_error(DP_ERR_SHAPE, "nloc too large");
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
  P.nloc = nloc;
  P.nnei = nnei;
  P.ntypes = ntypes;
  P.M1 = M1;
  P.pair_stride = g.nint * M1 * 6;
  for (int b = 0; b < DP_MAX_TYPES; ++b) P.sel[b] = seg.sel[b];
  P.inv_nnei = (real)(1.0 / (double)nnei);
  const int ychunks = (nnei + kGradThreads - 1) / kGradThreads;
  if (ychunks > 65535) return set_error(DP_ERR_SHAPE, "nnei = %d too large", nnei);
  const size_t smem = (size_t)4 * M1 * sizeof(real);
  dim3 grid((unsigned)nloc, (unsigned)ychunks);
  grad_kernel<real><<<grid, kGradThreads, smem, (cudaStream_t)stream>>>(P);
  return launch_status("dp_tabulate_fusion_grad");
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

}  // extern "C"
