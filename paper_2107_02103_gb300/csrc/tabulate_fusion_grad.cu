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
// Each thread gathers its own interval's coefficient row, which walks
// contiguous memory as m advances; dT_i is read through the read-only cache
// (every lane of an atom reads the same address).  Threads past the valid
// rows zero-fill the padding rows, packed the same way.
#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kGradThreads = 128;
constexpr int kGradChunk = 16;  // atoms whose valid rows are packed together

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
      ld6(cp + m * 6, cf);
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
  const int64_t ychunks = ((int64_t)kGradChunk * nnei + kGradThreads - 1) / kGradThreads;
  if (ychunks > 65535) return set_error(DP_ERR_SHAPE, "nnei = %d too large", nnei);
  const int64_t xchunks = (nloc + kGradChunk - 1) / kGradChunk;
  dim3 grid((unsigned)xchunks, (unsigned)ychunks);
  grad_kernel<real><<<grid, kGradThreads, 0, (cudaStream_t)stream>>>(P);
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
