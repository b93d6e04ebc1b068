// Compression step (Sec. II): the embedding net and its first two
// derivatives at the table nodes, and the six quintic coefficients of every
// interval and channel.  Setup work, run once per model.
#include "dp_common.cuh"

namespace dpc {

namespace {

constexpr int kNodeThreads = 128;
constexpr int kBuildThreads = 256;

struct NetDims {
  int32_t nlayer;
  int32_t maxw;
  int32_t w[DP_MAX_LAYERS + 1];
  int64_t P;  // parameters per pair
};

// One block per (node l, pair p).  Layer by layer in shared memory, with the
// d/dx and d2/dx2 of every activation carried alongside (forward mode):
//   z' = v' W, z'' = v'' W, h = tanh z, h' = (1 - h^2) z', h'' = (1 - h^2) z'' - 2 h (1 - h^2) z'^2,
// and the residual skip u = h + v (same width) or u = h + (v, v) (doubled width).
__global__ void __launch_bounds__(kNodeThreads) net_nodes_kernel(const double *__restrict__ params, NetDims nd,
                                                                 TableGeom g, double *__restrict__ y,
                                                                 double *__restrict__ dy, double *__restrict__ d2y) {
  extern __shared__ double sh[];
  const int l = blockIdx.x, p = blockIdx.y;
  double *v = sh, *v1 = sh + nd.maxw, *v2 = sh + 2 * nd.maxw;
  double *u = sh + 3 * nd.maxw, *u1 = sh + 4 * nd.maxw, *u2 = sh + 5 * nd.maxw;
  if (threadIdx.x == 0) {
    v[0] = node_x(g, l);
    v1[0] = 1.0;
    v2[0] = 0.0;
  }
  __syncthreads();
  const double *pp = params + (size_t)p * nd.P;
  for (int layer = 0; layer < nd.nlayer; ++layer) {
    const int a = nd.w[layer], b = nd.w[layer + 1];
    const double *W = pp, *bias = pp + (size_t)a * b;
    pp += (size_t)a * b + b;
    for (int o = threadIdx.x; o < b; o += blockDim.x) {
      double z = bias[o], z1 = 0.0, z2 = 0.0;
      for (int q = 0; q < a; ++q) {
        const double wv = W[(size_t)q * b + o];
        z = fma(v[q], wv, z);
        z1 = fma(v1[q], wv, z1);
        z2 = fma(v2[q], wv, z2);
      }
      const double h = tanh(z);
      const double sech2 = fma(-h, h, 1.0);
      const double h1 = sech2 * z1;
      const double h2 = sech2 * z2 - 2.0 * h * sech2 * z1 * z1;
      double s0 = 0.0, s1 = 0.0, s2 = 0.0;
      if (b == a || b == 2 * a) {
        const int src = o < a ? o : o - a;
        s0 = v[src];
        s1 = v1[src];
        s2 = v2[src];
      }
      u[o] = h + s0;
      u1[o] = h1 + s1;
      u2[o] = h2 + s2;
    }
    __syncthreads();
    double *t0 = v, *t1 = v1, *t2 = v2;
    v = u; v1 = u1; v2 = u2;
    u = t0; u1 = t1; u2 = t2;
  }
  const int M1 = nd.w[nd.nlayer];
  const size_t base = ((size_t)p * (g.nint + 1) + l) * M1;
  for (int m = threadIdx.x; m < M1; m += blockDim.x) {
    y[base + m] = v[m];
    dy[base + m] = v1[m];
    d2y[base + m] = v2[m];
  }
}

// ---- double-double arithmetic (Knuth's TwoSum, Dekker's product via fma)
struct dd {
  double hi, lo;
};
__device__ __forceinline__ dd two_sum(double a, double b) {
  const double s = a + b, bb = s - a;
  return {s, (a - (s - bb)) + (b - bb)};
}
__device__ __forceinline__ dd fast_two_sum(double a, double b) {
  const double s = a + b;
  return {s, b - (s - a)};
}
__device__ __forceinline__ dd two_prod(double a, double b) {
  const double p = a * b;
  return {p, fma(a, b, -p)};
}
__device__ __forceinline__ dd dd_add(dd x, dd y) {
  dd s = two_sum(x.hi, y.hi);
  const dd t = two_sum(x.lo, y.lo);
  s.lo += t.hi;
  s = fast_two_sum(s.hi, s.lo);
  s.lo += t.lo;
  return fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ dd dd_mul_d(dd x, double b) {
  dd p = two_prod(x.hi, b);
  p.lo = fma(x.lo, b, p.lo);
  return fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ dd dd_mul(dd x, dd y) {
  dd p = two_prod(x.hi, y.hi);
  p.lo = fma(x.hi, y.lo, fma(x.lo, y.hi, p.lo));
  return fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ double dd_val(dd x) { return x.hi + x.lo; }

// One thread per (pair, interval, channel).  Coefficients of
// g(t) = a t^5 + b t^4 + c t^3 + d t^2 + e t + f on [x_l, x_{l+1}) from the
// paper's closed forms (Sec. II), with h = y1 - y0 and Dt the interval width:
//   a = [12h - 6(y1' + y0')Dt + (y1'' - y0'')Dt^2] / (2 Dt^5)
//   b = [-30h + (14y1' + 16y0')Dt + (3y0'' - 2y1'')Dt^2] / (2 Dt^4)
//   c = [20h - (8y1' + 12y0')Dt - (3y0'' - y1'')Dt^2] / (2 Dt^3)
//   d = y0''/2, e = y0', f = y0.
// The brackets cancel down to O(Dt^5 |y^(5)|); they are formed in
// double-double so their rounding does not swamp what is left.
template <typename real>
__global__ void __launch_bounds__(kBuildThreads)
    table_build_kernel(const double *__restrict__ y, const double *__restrict__ dy, const double *__restrict__ d2y,
                       int npair, int M1, TableGeom g, real *__restrict__ table) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)npair * g.nint * M1;
  if (tid >= total) return;
  const int m = (int)(tid % M1);
  const int64_t pl = tid / M1;
  const int l = (int)(pl % g.nint);
  const int p = (int)(pl / g.nint);
  const size_t i0 = ((size_t)p * (g.nint + 1) + l) * M1 + m, i1 = i0 + M1;
  const double y0 = y[i0], y1 = y[i1], p0 = dy[i0], p1 = dy[i1], q0 = d2y[i0], q1 = d2y[i1];
  const double Dt = l < g.n0 ? g.stride0 : g.stride1;

  const dd h = two_sum(y1, -y0);
  const dd Dt2 = two_prod(Dt, Dt);
  // a
  const dd pa = dd_mul_d(two_sum(p1, p0), Dt);
  const dd qa = dd_mul(two_sum(q1, -q0), Dt2);
  const dd ba = dd_add(dd_add(dd_mul_d(h, 12.0), dd_mul_d(pa, -6.0)), qa);
  // b
  const dd pb = dd_mul_d(dd_add(two_prod(p1, 14.0), two_prod(p0, 16.0)), Dt);
  const dd qb = dd_mul(dd_add(two_prod(q0, 3.0), two_prod(q1, -2.0)), Dt2);
  const dd bb = dd_add(dd_add(dd_mul_d(h, -30.0), pb), qb);
  // c
  const dd pc = dd_mul_d(dd_add(two_prod(p1, 8.0), two_prod(p0, 12.0)), Dt);
  const dd qc = dd_mul(dd_add(two_prod(q0, 3.0), dd{-q1, 0.0}), Dt2);
  const dd bc = dd_add(dd_add(dd_mul_d(h, 20.0), dd_mul_d(pc, -1.0)), dd_mul_d(qc, -1.0));

  const double Dt3 = Dt * Dt * Dt, Dt4 = Dt3 * Dt, Dt5 = Dt4 * Dt;
  // pair-planar block of interval (p, l): [3][M1][2] = (a, b), (c, d), (e, f) planes
  real *blk = table + (size_t)pl * 6 * M1 + 2 * m;
  blk[0] = dcvt<real>(dd_val(ba) / (2.0 * Dt5));
  blk[1] = dcvt<real>(dd_val(bb) / (2.0 * Dt4));
  blk[2 * M1] = dcvt<real>(dd_val(bc) / (2.0 * Dt3));
  blk[2 * M1 + 1] = dcvt<real>(0.5 * q0);
  blk[4 * M1] = dcvt<real>(p0);
  blk[4 * M1 + 1] = dcvt<real>(y0);
}

template <typename real>
int table_build(const double *y, const double *dy, const double *d2y, int npair, int M1, const dp_table_info *info,
                real *table, void *stream) {
  clear_error();
  if (!y || !dy || !d2y || !table) return set_error(DP_ERR_NULL, "a required device pointer is NULL");
  if (npair < 1 || M1 < 1) return set_error(DP_ERR_SHAPE, "npair = %d and M1 = %d must be >= 1", npair, M1);
  TableGeom g;
  int rc = make_geom(info, &g);
  if (rc) return rc;
  const int64_t total = (int64_t)npair * g.nint * M1;
  if ((double)total * 6.0 >= 9.0e18) return set_error(DP_ERR_SHAPE, "table too large");
  const int64_t blocks = (total + kBuildThreads - 1) / kBuildThreads;
  table_build_kernel<real><<<(unsigned)blocks, kBuildThreads, 0, (cudaStream_t)stream>>>(y, dy, d2y, npair, M1, g,
                                                                                         table);
  return launch_status("dp_table_build");
}

}  // namespace

}  // namespace dpc

extern "C" {

int dp_embedding_net_nodes_f64(const double *params, const int32_t *widths, int nlayer, int npair,
                               const dp_table_info *info, double *y, double *dy, double *d2y, void *stream) {
  using namespace dpc;
  clear_error();
  if (!params || !widths || !y || !dy || !d2y) return set_error(DP_ERR_NULL, "a required pointer is NULL");
  if (npair < 1) return set_error(DP_ERR_SHAPE, "npair = %d < 1", npair);
  if (nlayer < 1 || nlayer > DP_MAX_LAYERS)
    return set_error(DP_ERR_UNSUPPORTED, "nlayer = %d outside [1, %d]", nlayer, DP_MAX_LAYERS);
  NetDims nd;
  nd.nlayer = nlayer;
  nd.maxw = 1;
  nd.P = 0;
  for (int l = 0; l <= DP_MAX_LAYERS; ++l) nd.w[l] = 0;
  for (int l = 0; l <= nlayer; ++l) {
    if (widths[l] < 1) return set_error(DP_ERR_SHAPE, "widths[%d] = %d < 1", l, widths[l]);
    if (widths[l] > DP_MAX_WIDTH) return set_error(DP_ERR_UNSUPPORTED, "widths[%d] = %d > %d", l, widths[l], DP_MAX_WIDTH);
    nd.w[l] = widths[l];
    if (widths[l] > nd.maxw) nd.maxw = widths[l];
  }
  if (widths[0] != 1) return set_error(DP_ERR_SHAPE, "widths[0] = %d, the embedding net has one input", widths[0]);
  for (int l = 0; l < nlayer; ++l) nd.P += (int64_t)widths[l] * widths[l + 1] + widths[l + 1];
  TableGeom g;
  const int rc = make_geom(info, &g);
  if (rc) return rc;
  const size_t smem = (size_t)6 * nd.maxw * sizeof(double);
  if (smem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(net_nodes_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "dp_embedding_net_nodes: %s", cudaGetErrorString(e));
  }
  dim3 grid((unsigned)(g.nint + 1), (unsigned)npair);
  net_nodes_kernel<<<grid, kNodeThreads, smem, (cudaStream_t)stream>>>(params, nd, g, y, dy, d2y);
  return launch_status("dp_embedding_net_nodes");
}

int dp_table_build_f64(const double *y, const double *dy, const double *d2y, int npair, int M1,
                       const dp_table_info *info, double *table, void *stream) {
  return dpc::table_build<double>(y, dy, d2y, npair, M1, info, table, stream);
}

int dp_table_build_f32(const double *y, const double *dy, const double *d2y, int npair, int M1,
                       const dp_table_info *info, float *table, void *stream) {
  return dpc::table_build<float>(y, dy, d2y, npair, M1, info, table, stream);
}

int dp_table_build_df64(const double *y, const double *dy, const double *d2y, int npair, int M1,
                        const dp_table_info *info, float *table, void *stream) {
  return dpc::table_build<dpc::df64>(y, dy, d2y, npair, M1, info, reinterpret_cast<dpc::df64 *>(table), stream);
}

}  // extern "C"
