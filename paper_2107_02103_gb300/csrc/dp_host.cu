// Host-side pieces of the C ABI: error state, table-range rules, argument
// validation.  No device code.
#include <cstdarg>
#include <cstdio>
#include <string>

#include "dp_common.cuh"

namespace dpc {

static thread_local std::string g_error;

int set_error(int code, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_error = buf;
  return code;
}

void clear_error() { g_error.clear(); }

int launch_status(const char *what) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return set_error(DP_ERR_CUDA, "%s: launch failed: %s", what, cudaGetErrorString(e));
  return DP_OK;
}

// Kernel timing hook (off unless dp_profile_begin was called): calls that launch several kernels
// record the caller's events on their stream, one after each kernel, in order, with the kernel's name.
namespace {
constexpr int kMaxProfileEvents = 4096;
struct Profile {
  cudaEvent_t ev[kMaxProfileEvents];
  const char *name[kMaxProfileEvents];
  int n = 0, cap = 0;
  bool on = false;
};
Profile g_prof;
}  // namespace

void prof_mark(const char *name, cudaStream_t st) {
  if (!g_prof.on || g_prof.n >= g_prof.cap) return;
  if (cudaEventRecord(g_prof.ev[g_prof.n], st) == cudaSuccess) g_prof.name[g_prof.n++] = name;
}

static bool finite(double x) { return std::isfinite(x); }

int make_geom(const dp_table_info *info, TableGeom *g) {
  if (!info) return set_error(DP_ERR_NULL, "table info is NULL");
  const dp_table_info &in = *info;
  if (!finite(in.lower) || !finite(in.upper) || !finite(in.upper_ext) || !finite(in.stride0) ||
      !finite(in.stride1))
    return set_error(DP_ERR_TABLE_INFO, "table info has a non-finite field");
  if (!(in.stride0 > 0.0) || !(in.stride1 > 0.0))
    return set_error(DP_ERR_TABLE_INFO, "table strides must be positive (%g, %g)", in.stride0, in.stride1);
  if (!(in.upper > in.lower) || !(in.upper_ext >= in.upper))
    return set_error(DP_ERR_TABLE_INFO, "table range needs lower < upper <= upper_ext (%g, %g, %g)", in.lower,
                     in.upper, in.upper_ext);
  const double r0 = (in.upper - in.lower) / in.stride0;
  const double r1 = (in.upper_ext - in.upper) / in.stride1;
  const long long n0 = std::llround(r0), n1 = std::llround(r1);
  if (n0 < 1 || std::fabs(r0 - (double)n0) > 1e-9 * (n0 > 1 ? (double)n0 : 1.0))
    return set_error(DP_ERR_TABLE_INFO, "(upper - lower)/stride0 = %.17g is not a positive integer", r0);
  if (n1 < 0 || std::fabs(r1 - (double)n1) > 1e-9 * (n1 > 1 ? (double)n1 : 1.0))
    return set_error(DP_ERR_TABLE_INFO, "(upper_ext - upper)/stride1 = %.17g is not an integer", r1);
  if (n0 + n1 > (1LL << 24)) return set_error(DP_ERR_TABLE_INFO, "table has %lld intervals (limit 2^24)", n0 + n1);
  g->lower = in.lower;
  g->upper = in.upper;
  g->upper_ext = in.upper_ext;
  g->stride0 = in.stride0;
  g->stride1 = in.stride1;
  g->inv0 = 1.0 / in.stride0;
  g->inv1 = 1.0 / in.stride1;
  g->n0 = (int32_t)n0;
  g->n1 = (int32_t)n1;
  g->nint = (int32_t)(n0 + n1);
  return DP_OK;
}

int make_segments(int ntypes, const int32_t *sel, int nnei, Segments *out) {
  if (!sel) return set_error(DP_ERR_NULL, "sel is NULL");
  if (ntypes < 1) return set_error(DP_ERR_SHAPE, "ntypes = %d < 1", ntypes);
  if (ntypes > DP_MAX_TYPES) return set_error(DP_ERR_UNSUPPORTED, "ntypes = %d > %d", ntypes, DP_MAX_TYPES);
  if (nnei < 1) return set_error(DP_ERR_SHAPE, "nnei = %d < 1", nnei);
  long long sum = 0;
  for (int b = 0; b < DP_MAX_TYPES; ++b) out->sel[b] = 0;
  for (int b = 0; b < ntypes; ++b) {
    if (sel[b] < 0) return set_error(DP_ERR_SHAPE, "sel[%d] = %d < 0", b, sel[b]);
    out->sel[b] = sel[b];
    sum += sel[b];
  }
  if (sum != nnei) return set_error(DP_ERR_SHAPE, "sum(sel) = %lld != nnei = %d", sum, nnei);
  out->ntypes = ntypes;
  out->nnei = nnei;
  return DP_OK;
}

int check_fusion_args(const void *table, const dp_table_info *info, const void *s, const void *Rt, int64_t nloc,
                      int nnei, int ntypes, const int32_t *sel, int M1, const void *out0, const void *out1,
                      TableGeom *g, Segments *seg) {
  if (nloc < 0) return set_error(DP_ERR_SHAPE, "nloc = %lld < 0", (long long)nloc);
  if (nloc > 0 && (!table || !s || !Rt || !out0 || !out1))
    return set_error(DP_ERR_NULL, "a required device pointer is NULL");
  if (M1 < 1) return set_error(DP_ERR_SHAPE, "M1 = %d < 1", M1);
  if (M1 > DP_MAX_M1) return set_error(DP_ERR_UNSUPPORTED, "M1 = %d > %d", M1, DP_MAX_M1);
  int rc = make_segments(ntypes, sel, nnei, seg);
  if (rc) return rc;
  rc = make_geom(info, g);
  if (rc) return rc;
  const double elems = (double)ntypes * ntypes * g->nint * (double)M1 * 6.0;
  if (elems >= 2147483647.0) return set_error(DP_ERR_SHAPE, "table of %.0f elements exceeds 2^31", elems);
  return DP_OK;
}

}  // namespace dpc

extern "C" {

const char *dp_last_error(void) { return dpc::g_error.c_str(); }

int dp_profile_begin(void *const *events, int n) {
  dpc::clear_error();
  if (n < 0 || n > dpc::kMaxProfileEvents)
    return dpc::set_error(DP_ERR_SHAPE, "dp_profile_begin: n = %d outside [0, %d]", n, dpc::kMaxProfileEvents);
  if (n > 0 && !events) return dpc::set_error(DP_ERR_NULL, "dp_profile_begin: events is NULL");
  for (int i = 0; i < n; ++i) {
    if (!events[i]) return dpc::set_error(DP_ERR_NULL, "dp_profile_begin: events[%d] is NULL", i);
    dpc::g_prof.ev[i] = static_cast<cudaEvent_t>(events[i]);
  }
  dpc::g_prof.n = 0;
  dpc::g_prof.cap = n;
  dpc::g_prof.on = n > 0;
  return DP_OK;
}

int dp_profile_end(void) {
  dpc::g_prof.on = false;
  return dpc::g_prof.n;
}

const char *dp_profile_name(int i) { return i >= 0 && i < dpc::g_prof.n ? dpc::g_prof.name[i] : ""; }

int dp_tc_wait_timeouts(unsigned int *count) {
  dpc::clear_error();
  if (!count) return dpc::set_error(DP_ERR_NULL, "dp_tc_wait_timeouts: count is NULL");
  *count = 0;
  int rc = dpc::take_wait_timeouts_tabulate(count);
  if (!rc) rc = dpc::take_wait_timeouts_fitting(count);
  return rc;
}

int dp_table_info_make(double s_min, double s_max, double stride0, double stride1, double ext, dp_table_info *out) {
  dpc::clear_error();
  if (!out) return dpc::set_error(DP_ERR_NULL, "out is NULL");
  if (!std::isfinite(s_min) || !std::isfinite(s_max) || !(s_max > 0.0) || !(s_min <= s_max))
    return dpc::set_error(DP_ERR_TABLE_INFO, "data range [%g, %g] must be finite with s_max > 0", s_min, s_max);
  if (!(stride0 > 0.0) || !(stride1 > 0.0) || !(ext >= 1.0) || !std::isfinite(ext))
    return dpc::set_error(DP_ERR_TABLE_INFO, "need stride0 > 0, stride1 > 0, ext >= 1");
  const double ratio = stride1 / stride0;
  if (std::fabs(ratio - std::nearbyint(ratio)) > 1e-9 * ratio)
    return dpc::set_error(DP_ERR_TABLE_INFO, "stride1/stride0 = %.17g must be an integer", ratio);
  dp_table_info in;
  in.stride0 = stride0;
  in.stride1 = stride1;
  in.lower = s_min >= 0.0 ? 0.0 : stride0 * std::floor(s_min / stride0);
  in.upper = stride1 * std::ceil(s_max / stride1);
  in.upper_ext = ext * in.upper;
  dpc::TableGeom g;
  const int rc = dpc::make_geom(&in, &g);
  if (rc) return rc;
  *out = in;
  return DP_OK;
}

int dp_table_info_sizes(const dp_table_info *info, int32_t *n0, int32_t *n1) {
  dpc::clear_error();
  if (!n0 || !n1) return dpc::set_error(DP_ERR_NULL, "n0/n1 is NULL");
  dpc::TableGeom g;
  const int rc = dpc::make_geom(info, &g);
  if (rc) return rc;
  *n0 = g.n0;
  *n1 = g.n1;
  return DP_OK;
}

}  // extern "C"
