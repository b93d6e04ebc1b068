/*
 * dp_compress.h -- C ABI of the GB300 (sm_103a) DP Compress tabulate-fusion library.
 *
 * The library implements the compressed single-atom workflow of DP Compress
 * (Lu et al., arXiv 2107.02103, Sec. II "Methods"): the embedding net G(s) is
 * replaced by piecewise fifth-order polynomials on a uniform grid, and the
 * product S_i = G_i^T R~_i (here T_i = S_i^T / N_c, 4 x M) is formed in one
 * fused pass that never stores G_i and skips padded neighbour rows.
 *
 * Conventions shared by every entry point
 *   - Every pointer argument to a *_f64 / *_f32 compute call is DEVICE memory
 *     allocated and owned by the caller, unless marked "host".  The library
 *     allocates nothing and keeps no pointer after returning.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  Calls only ENQUEUE work on it; they never synchronise.  A
 *     non-zero status means nothing was enqueued, except DP_ERR_CUDA from a
 *     failed launch.  Faults during execution surface at the caller's next
 *     synchronisation on that stream.
 *   - Outputs are fully overwritten (padding rows included); nothing needs to
 *     be zeroed beforehand.  Inputs and outputs must not overlap.
 *   - Arrays are C-contiguous (row-major) in the layouts given per argument.
 *     Device pointers must be 16-byte aligned (any cudaMalloc / torch
 *     allocation is).
 *   - Return value: DP_OK (0) or a negative dp_status; dp_last_error()
 *     then describes the failure (per calling thread).
 *
 * Notation: nloc atoms, ntypes atom types, sel[b] rows reserved for
 * neighbours of type b, nnei = N_c = sum_b sel[b] rows per atom; rows of
 * type b occupy [off_b, off_b + sel[b]) with off_b = sum_{c<b} sel[c]; the
 * first nvalid[i][b] of them are real neighbours, the rest are zero padding
 * (Sec. II: neighbours sorted by type, then distance; missing rows are 0).
 * M1 = M embedding channels, M2 = M' < M leading channels of the descriptor.
 * A type pair (alpha, beta) = (centre type, neighbour type) has its own table
 * at index alpha * ntypes + beta.
 */
#ifndef DP_COMPRESS_H
#define DP_COMPRESS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DP_MAX_TYPES 8     /* ntypes <= DP_MAX_TYPES                         */
#define DP_MAX_M1 256      /* fused forward supports M1 <= DP_MAX_M1          */
#define DP_MAX_WIDTH 1024  /* embedding-net layer width limit                */
#define DP_MAX_LAYERS 8    /* embedding-net depth limit                      */

/*
 * Table range (Sec. II: the domain of the embedding input is cut into equal
 * intervals; its bounds come from a scan of the data, the upper bound
 * covering the largest value).  Fine segment [lower, upper) with step
 * stride0, coarse extrapolation segment [upper, upper_ext) with step stride1.
 * Derived: n0 = (upper - lower) / stride0 and n1 = (upper_ext - upper) /
 * stride1, both integral within 1e-9; nint = n0 + n1 intervals; nodes
 * x_l = lower + l*stride0 (l < n0), x_n0 = upper, x_{n0+k} = upper + k*stride1.
 */
typedef struct dp_table_info {
  double lower;
  double upper;
  double upper_ext;
  double stride0;
  double stride1;
} dp_table_info;

typedef enum dp_status {
  DP_OK = 0,
  DP_ERR_NULL = -1,        /* a required pointer is NULL                        */
  DP_ERR_SHAPE = -2,       /* a size is negative, inconsistent or too large     */
  DP_ERR_TABLE_INFO = -3,  /* table range not positive / not integral in steps  */
  DP_ERR_CUDA = -4,        /* a CUDA launch failed (message has the CUDA error) */
  DP_ERR_UNSUPPORTED = -5  /* outside the limits above (M1, ntypes, width)      */
} dp_status;

/* Message for the last non-OK status returned on the calling thread ("" if none).
   The string stays valid until the next library call on that thread. */
const char *dp_last_error(void);

/*
 * Host-only.  Table range from the data range [s_min, s_max] (Sec. II, the
 * range is set by scanning the data; the upper bound covers its maximum):
 *   lower = 0 if s_min >= 0 else stride0 * floor(s_min / stride0)
 *   upper = stride1 * ceil(s_max / stride1),  upper_ext = ext * upper.
 * Requires stride0 > 0, stride1 > 0, stride1/stride0 integral, ext >= 1,
 * s_max > 0, s_min <= s_max.  Writes *out (host).  DP_ERR_TABLE_INFO otherwise.
 */
int dp_table_info_make(double s_min, double s_max, double stride0, double stride1, double ext,
                       dp_table_info *out);

/* Host-only.  Validates *info and writes n0, n1 (host) -- see dp_table_info. */
int dp_table_info_sizes(const dp_table_info *info, int32_t *n0, int32_t *n1);

/*
 * Embedding net at the table nodes (Sec. II: the value y_l = G_m(x_l) and the
 * derivatives y'_l, y''_l at every interpolation point, which the paper notes
 * can be evaluated efficiently).  Net of `nlayer` layers with widths
 * widths[0..nlayer] (host array, widths[0] == 1, widths[nlayer] == M1): layer
 * l maps v (width a) to u (width b) by z = v W_l + b_l, h = tanh(z) and
 *   u = h + v (b == a),  u = h + (v, v) (b == 2a),  u = h (otherwise).
 *   params  [npair][P] f64, per pair and layer W_l [a][b] row-major then b_l [b],
 *           P = sum_l (a_l b_l + b_l).
 *   y, dy, d2y  [npair][nint + 1][M1] f64 outputs: G, dG/dx, d2G/dx2 at x_l.
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (npair < 1, widths[0] != 1),
 * DP_ERR_UNSUPPORTED (nlayer > DP_MAX_LAYERS, width > DP_MAX_WIDTH),
 * DP_ERR_TABLE_INFO, DP_ERR_CUDA.
 */
int dp_embedding_net_nodes_f64(const double *params, const int32_t *widths, int nlayer, int npair,
                               const dp_table_info *info, double *y, double *dy, double *d2y, void *stream);

/*
 * Quintic Hermite table (Sec. II: on interval l, g_m^l(t) = a t^5 + b t^4 +
 * c t^3 + d t^2 + e t + f with t = x - x_l, and the closed forms of a..f
 * from (y, y', y'') at x_l and x_{l+1}, h = y_{l+1} - y_l, Dt = x_{l+1} - x_l).
 * The brackets of a, b, c are evaluated in double-double arithmetic (they
 * cancel to O(Dt^5) relative) and rounded once.
 *   y, dy, d2y  [npair][nint + 1][M1] f64 node values (device).
 *   table       [npair][nint][3][M1][2], f64 or rounded to f32: per interval a
 *               pair-planar block -- the (a, b) pairs of channels 0..M1-1, then
 *               the (c, d) pairs, then the (e, f) pairs -- so that lanes reading
 *               consecutive channels make fully coalesced loads.
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (npair < 1, M1 < 1), DP_ERR_TABLE_INFO,
 * DP_ERR_CUDA.
 */
int dp_table_build_f64(const double *y, const double *dy, const double *d2y, int npair, int M1,
                       const dp_table_info *info, double *table, void *stream);
int dp_table_build_f32(const double *y, const double *dy, const double *d2y, int npair, int M1,
                       const dp_table_info *info, float *table, void *stream);

/*
 * Fused tabulated embedding + contraction, forward (Sec. II, kernel fusion:
 * the column of G_i^T for neighbour j is evaluated from the table in
 * registers and immediately multiplied into R~_i, only for valid j):
 *   T[i][k][m] = (1/nnei) * sum_b sum_{j < nvalid[i][b]} R~[i][off_b + j][k] * g_m(s[i][off_b + j])
 * with g_m the table of pair (atype[i], b).  Interval search: s in [lower,
 * upper) uses l = floor((s - lower)/stride0), s in [upper, upper_ext) uses
 * n0 + floor((s - upper)/stride1); s < lower evaluates the first node, s >=
 * upper_ext the last node; NaN s gives NaN in that atom's T.
 *   table   [npair][nint][3][M1][2] (from dp_table_build_*), npair = ntypes^2
 *   s       [nloc][nnei]      embedding input per row
 *   Rt      [nloc][nnei][4]   environment-matrix rows
 *   nvalid  [nloc][ntypes] int32, real rows per type segment; entries are
 *           clamped into [0, sel[b]] (rows beyond are never read);
 *           NULL = every row valid
 *   atype   [nloc] int32 centre type, clamped into [0, ntypes); NULL = type 0
 *   sel     [ntypes] int32 HOST array; nnei must equal sum(sel)
 *   T       [nloc][4][M1] output
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (nloc < 0, nnei < 1, sum(sel) != nnei,
 * M1 < 1, table larger than 2^31 elements), DP_ERR_UNSUPPORTED (ntypes >
 * DP_MAX_TYPES, M1 > DP_MAX_M1), DP_ERR_TABLE_INFO, DP_ERR_CUDA.  nloc == 0
 * enqueues nothing, reads no device pointer (they may be NULL) and returns
 * DP_OK once the sizes and the table info are valid.
 */
int dp_tabulate_fusion_fwd_f64(const double *table, const dp_table_info *info, const double *s, const double *Rt,
                               const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                               const int32_t *sel, int M1, double *T, void *stream);
int dp_tabulate_fusion_fwd_f32(const float *table, const dp_table_info *info, const float *s, const float *Rt,
                               const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                               const int32_t *sel, int M1, float *T, void *stream);

/*
 * The same forward by interval moments.  Neighbours are sorted by distance
 * inside a type segment (Sec. II), so consecutive valid rows often fall in
 * the same table interval l.  For such a run the per-neighbour sum regroups
 * exactly as
 *   sum_{j in run} R~_j[k] g_m(t_j) = sum_q C_{l,m,q} W[k][q],   W[k][q] = sum_{j in run} R~_j[k] t_j^q,
 * with C_{l,m,q} the t^q coefficient: 24 FMA per channel per run instead of
 * 9 per channel per neighbour.  Runs of 3 or more rows go this way, shorter
 * ones neighbour by neighbour.  Same arguments, results and errors as
 * dp_tabulate_fusion_fwd_* (equal up to rounding order).
 */
int dp_tabulate_fusion_fwd_moments_f64(const double *table, const dp_table_info *info, const double *s,
                                       const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                       int nnei, int ntypes, const int32_t *sel, int M1, double *T, void *stream);
int dp_tabulate_fusion_fwd_moments_f32(const float *table, const dp_table_info *info, const float *s,
                                       const float *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                       int nnei, int ntypes, const int32_t *sel, int M1, float *T, void *stream);

/*
 * Forward and descriptor in one pass (Sec. II: T_i, then D_i = S_i (S_i^<)^T
 * with S_i = T_i^T): the same T as dp_tabulate_fusion_fwd_* and
 *   D[i][m][n] = sum_k T[i][k][m] * T[i][k][n],  n < M2,
 * formed while T_i is still on chip (no second read of T).  Arguments as
 * dp_tabulate_fusion_fwd_* plus M2 and D [nloc][M1][M2] (output).
 * Extra errors: DP_ERR_SHAPE (M2 < 1 or M2 > M1), DP_ERR_UNSUPPORTED (M2 > 32).
 */
int dp_tabulate_fusion_fwd_descriptor_f64(const double *table, const dp_table_info *info, const double *s,
                                          const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                          int nnei, int ntypes, const int32_t *sel, int M1, int M2, double *T,
                                          double *D, void *stream);
int dp_tabulate_fusion_fwd_descriptor_f32(const float *table, const dp_table_info *info, const float *s,
                                          const float *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                          int nnei, int ntypes, const int32_t *sel, int M1, int M2, float *T,
                                          float *D, void *stream);

/*
 * Backward of the fused forward (Sec. II: the compressed model serves both
 * the forward and the backward propagation, which yields forces and virials).
 * Given dT = dE/dT_i:
 *   dRt[i][row][k] = (1/nnei) * sum_m dT[i][k][m] * g_m(s_row)
 *   ds[i][row]     = (1/nnei) * sum_m (sum_k dT[i][k][m] * R~[i][row][k]) * g'_m(s_row)
 * for valid rows; g' = 0 where s was clamped to an end node; padding rows
 * get ds = 0 and dRt = 0.  When s is the first column of R~ the total
 * derivative for that column is ds + dRt[..][0].
 *   dT   [nloc][4][M1] input;  ds [nloc][nnei], dRt [nloc][nnei][4] outputs.
 *   Other arguments, limits and errors as dp_tabulate_fusion_fwd_*.
 */
int dp_tabulate_fusion_grad_f64(const double *table, const dp_table_info *info, const double *s, const double *Rt,
                                const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                const int32_t *sel, int M1, const double *dT, double *ds, double *dRt,
                                void *stream);
int dp_tabulate_fusion_grad_f32(const float *table, const dp_table_info *info, const float *s, const float *Rt,
                                const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                const int32_t *sel, int M1, const float *dT, float *ds, float *dRt, void *stream);

/*
 * The same backward by interval moments.  For a run of consecutive valid
 * rows in one table interval l (rows are sorted by distance inside a type
 * segment, Sec. II), with C_{l,m,q} the t^q coefficient of g_m on l,
 *   H[k][q] = sum_m dT[i][k][m] C_{l,m,q}
 * is formed once per run (24 FMA per channel), and each row follows from it:
 *   dRt[i][row][k] = (1/nnei) sum_q t^q H[k][q]
 *   ds[i][row]     = (1/nnei) sum_k R~[i][row][k] sum_{q>=1} q t^(q-1) H[k][q]
 * (the channel sums of dp_tabulate_fusion_grad_* taken in the other order).
 * Same arguments, results, limits and errors as dp_tabulate_fusion_grad_*.
 */
int dp_tabulate_fusion_grad_moments_f64(const double *table, const dp_table_info *info, const double *s,
                                        const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                        int nnei, int ntypes, const int32_t *sel, int M1, const double *dT, double *ds,
                                        double *dRt, void *stream);
int dp_tabulate_fusion_grad_moments_f32(const float *table, const dp_table_info *info, const float *s,
                                        const float *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                        int nnei, int ntypes, const int32_t *sel, int M1, const float *dT, float *ds,
                                        float *dRt, void *stream);

/*
 * The f64 forward and backward with the per-interval contraction on the
 * tensor cores (tcgen05).  Same inputs, results, limits and errors as
 * dp_tabulate_fusion_fwd_f64 / dp_tabulate_fusion_grad_f64, with the table
 * replaced by a plan made from it once (dp_tabulate_tc_plan_f64) and a work
 * buffer.  With u = t / Delta_l in [0, 1] (Delta_l = stride0 on the fine
 * grid, stride1 on the coarse one) and c'_q = c_q Delta_l^q, the interval
 * moments of the rows of atom i,
 *   W[k][(b, l, q)] = sum_{valid rows j of segment b in interval l} R~[i][j][k] u_j^q,
 * turn the forward into a GEMM over K = (neighbour type b, interval l, q):
 *   T[i][k][m] = (1/nnei) sum_{(b, l, q)} W[k][(b, l, q)] c'_q(pair (atype[i], b), l, m),
 * and the backward into the transposed one, dW[k][(b, l, q)] =
 * (1/nnei) sum_m dT[i][k][m] c'_q(..., l, m), from which every valid row
 * takes dRt[i][j][k] = sum_q dW[k][(b, l, q)] u_j^q and ds[i][j] =
 * sum_k R~[i][j][k] sum_{q>=1} q dW[k][(b, l, q)] u_j^(q-1) / Delta_l (0
 * where s was clamped).  Both GEMMs run on digit-split operands with fp16
 * MMAs and exact fp32 sums, and round each output once to f64: the forward
 * as in dp_fitting_*_tc_f64 (nine balanced 6-bit digits per element, in
 * [-32, 32], scaled by the row's or column's power of two; at most 1792 of K
 * per partial sum; error below about K 2^-49 max|row| max|column|, K the
 * used intervals x 6), the backward, whose K is M1, in seven balanced 8-bit
 * digits (in [-128, 128]; error below K 2^-50 max|row| max|column|) while
 * M1 <= 144, else as the forward.  Only the intervals some atom of a 12-atom
 * (forward) or 8-atom (backward) tile uses enter its GEMM.  Rows need
 * not be sorted, though sorted rows (one run per interval) do the least
 * FP64 work.  NaN s gives NaN in that atom's T (forward) and in that row's
 * ds and dRt (backward); inf or NaN in dT gives NaN in the atom's rows.
 *
 * The forward also writes the descriptor when D is not NULL: D[i][m][n] =
 * sum_k T[i][k][m] T[i][k][n] for n < M2 (dp_descriptor_contract_f64,
 * computed from T in the same kernel that finishes T, with the same bits as
 * that call), D [nloc][M1][M2] on the device, 1 <= M2 <= M1 (else
 * DP_ERR_SHAPE).  With D NULL, M2 is ignored.
 *
 * The plan holds the scaled coefficients c'_q / nnei of every centre type
 * and their digit planes for both GEMMs; it depends only on the table, its
 * info, nnei, ntypes and M1, so a caller makes it once per table (it is
 * setup, like the table build) and passes it to every call.
 *   dp_tabulate_tc_plan_bytes  the size of its device buffer (0 on bad sizes).
 *   dp_tabulate_tc_plan_f64    fills `buf` (device, caller-owned, 256-byte
 *                              aligned, at least that many bytes) from the
 *                              table [ntypes*ntypes][nint][M1][6] (as
 *                              dp_table_build_f64 writes it), asynchronously
 *                              on `stream`, and the host record *plan (the
 *                              buffer, its size and the geometry it was made
 *                              for, which every call checks against its own
 *                              arguments: DP_ERR_SHAPE if they differ).  The
 *                              buffer must not change while calls use it.
 *   work, work_bytes  device scratch, caller-owned, 256-byte aligned, at
 *                     least dp_tabulate_tc_work_bytes(info, nloc, nnei,
 *                     ntypes, M1) bytes (one size for both directions): the
 *                     slot keys (int16, one per interval an atom uses), their
 *                     counts and the used-slice flags of every atom (kept
 *                     from the forward for the backward), and for one chunk
 *                     of at most 16416 atoms the moments or their gradients
 *                     per (atom, interval), the backward's B digit planes,
 *                     the forward's schedule and its partial results.
 *                     Calls sharing a work buffer must not overlap on the
 *                     GPU.
 *   flags (backward)  0, or DP_TC_REUSE_RUNS: the forward call on the same
 *                     plan, s, nvalid, atype, nloc and work buffer ran before
 *                     this call on the stream, and nothing has written the
 *                     work buffer or those inputs since; the backward then
 *                     takes the forward's slot keys and slice flags instead
 *                     of finding them again.  The library cannot check this
 *                     contract; broken, the results are wrong.
 * Extra errors: DP_ERR_NULL / DP_ERR_SHAPE for a missing, short or
 * misaligned work or plan buffer, or a plan made for another geometry;
 * DP_ERR_SHAPE for unknown flags; DP_ERR_UNSUPPORTED for more than 4096
 * intervals per centre type (ntypes x nint), whose per-atom key map would
 * not fit in shared memory.
 */
typedef struct dp_tc_plan {
  const void *data;   /* the plan's device buffer */
  size_t bytes;       /* its size */
  dp_table_info info; /* the geometry it was made for */
  int32_t nnei, ntypes, M1;
} dp_tc_plan;
#define DP_TC_REUSE_RUNS 1
size_t dp_tabulate_tc_plan_bytes(const dp_table_info *info, int nnei, int ntypes, int M1);
int dp_tabulate_tc_plan_f64(const double *table, const dp_table_info *info, int nnei, int ntypes, int M1, void *buf,
                            size_t bytes, dp_tc_plan *plan, void *stream);
size_t dp_tabulate_tc_work_bytes(const dp_table_info *info, int64_t nloc, int nnei, int ntypes,
                                 int M1); /* 0 on bad sizes or table info */
int dp_tabulate_fusion_fwd_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt,
                                  const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                  const int32_t *sel, int M1, double *T, int M2, double *D, void *work,
                                  size_t work_bytes, void *stream);
int dp_tabulate_fusion_grad_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *s, const double *Rt,
                                   const int32_t *nvalid, const int32_t *atype, int64_t nloc, int nnei, int ntypes,
                                   const int32_t *sel, int M1, const double *dT, double *ds, double *dRt, void *work,
                                   size_t work_bytes, int flags, void *stream);

/*
 * The same two calls with the environment matrix's front end and the force
 * back end fused in (Sec. II: s(r), the rows R~ and their normalisation;
 * the forces and virial by the chain rule), so that s, R~, ds and dR~ never
 * reach memory.  The rows are formed from coord [nall][3] and the neighbour
 * list nlist [nloc][nnei] (each type segment's neighbours first, -1 after)
 * exactly as dp_env_mat_f64 forms them, with the same env; the forward then
 * writes T (and D when D is not NULL, as dp_tabulate_fusion_fwd_tc_f64) and,
 * when nvalid is not NULL, the counts of rows with a neighbour [nloc][ntypes]
 * as dp_env_mat_f64 does.  The backward takes dT and adds what
 * dp_force_virial_f64 would add from the ds and dR~ that
 * dp_tabulate_fusion_grad_tc_f64 would write: F [nall][3] and virial [9],
 * both zeroed first (F holds the forces on the local atoms and the
 * reactions on the neighbours, ghosts included), up to the order of the
 * floating-point additions.  plan, work and flags as for the unfused calls
 * (DP_TC_REUSE_RUNS: the fused forward ran on the same plan, coord, nlist,
 * env, atype, nloc and work buffer).  Extra errors: DP_ERR_NULL for a missing
 * env, coord, nlist, F or virial; DP_ERR_TABLE_INFO for env out of range
 * (as dp_env_mat_f64); DP_ERR_SHAPE for nall < nloc.
 */
struct dp_env_info; /* defined with dp_env_mat_f64 below */
int dp_tabulate_fusion_env_fwd_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *coord,
                                      const int32_t *nlist, const struct dp_env_info *env, const int32_t *atype,
                                      int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M1,
                                      int32_t *nvalid, double *T, int M2, double *D, void *work, size_t work_bytes,
                                      void *stream);
int dp_tabulate_fusion_env_grad_tc_f64(const dp_tc_plan *plan, const dp_table_info *info, const double *coord,
                                       const int32_t *nlist, const struct dp_env_info *env, const int32_t *atype,
                                       int64_t nloc, int64_t nall, int nnei, int ntypes, const int32_t *sel, int M1,
                                       const double *dT, double *F, double *virial, void *work, size_t work_bytes,
                                       int flags, void *stream);

/*
 * Kernel timing hook, for profiling (off by default; not thread-safe: one
 * profiling session per process).  dp_profile_begin hands the library n
 * caller-created cudaEvent_t handles (as void*, created with timing enabled,
 * owned by the caller); until dp_profile_end, the calls that launch several
 * kernels (dp_tabulate_fusion_*_tc_f64) record the next event on their
 * stream when they start and after each of their kernels, so that the time
 * between consecutive events of one call is one kernel's.  dp_profile_name(i)
 * names what event i follows ("tc_fwd" / "tc_grad" for a call's start);
 * recording stops when the n events are used.  dp_profile_end turns the hook
 * off and returns how many events were recorded.  Errors: DP_ERR_SHAPE (n < 0
 * or n > 4096), DP_ERR_NULL.
 */
int dp_profile_begin(void *const *events, int n);
int dp_profile_end(void);
const char *dp_profile_name(int i);

/*
 * Diagnostic (not part of the paper's method): every wait of the tensor-core
 * GEMM kernels (dp_tabulate_fusion_*_tc_f64, dp_fitting_*_tc_f64) on an
 * mbarrier is bounded; a CTA whose wait gives up writes NaN outputs, reads
 * no accumulator and counts one timeout on the device.  This call waits for
 * the device to finish (cudaDeviceSynchronize), writes the count since the
 * last call to *count (host) and clears it.  0 in normal operation.
 * Errors: DP_ERR_NULL, DP_ERR_CUDA.
 */
int dp_tc_wait_timeouts(unsigned int *count);


/*
 * Descriptor (Sec. II): with S_i = T_i^T (M1 x 4) and S_i^< its first M2
 * rows, D_i = S_i (S_i^<)^T, i.e. D[i][m][n] = sum_k T[i][k][m] * T[i][k][n].
 *   T [nloc][4][M1] input,  D [nloc][M1][M2] output.
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (nloc < 0, M1 < 1, M2 < 1, M2 > M1),
 * DP_ERR_UNSUPPORTED (M1 > 4096, or T_i of four atoms not fitting in 227 KB
 * of shared memory: M1 > 1816 in f64, 3632 in f32), DP_ERR_CUDA.  nloc == 0
 * returns DP_OK without reading T or D.
 */
int dp_descriptor_contract_f64(const double *T, int64_t nloc, int M1, int M2, double *D, void *stream);
int dp_descriptor_contract_f32(const float *T, int64_t nloc, int M1, int M2, float *D, void *stream);

/*
 * Backward of the descriptor (Sec. II: D_i = S_i (S_i^<)^T is quadratic in
 * S_i = T_i^T; the backward propagation of the compressed model runs through
 * it before reaching the tabulated embedding).  Given dD = dE/dD:
 *   dT[i][k][m] = sum_{n<M2} dD[i][m][n] T[i][k][n] + [m < M2] sum_{m'} dD[i][m'][m] T[i][k][m']
 *   T [nloc][4][M1], dD [nloc][M1][M2] inputs;  dT [nloc][4][M1] output, fully
 *   overwritten (feed it to dp_tabulate_fusion_grad_*).
 * Errors, limits and the nloc == 0 rule as dp_descriptor_contract_*; the
 * backward stages T_i and dT_i (M1 > 908 in f64, 1816 in f32 is
 * DP_ERR_UNSUPPORTED).
 */
int dp_descriptor_contract_grad_f64(const double *T, const double *dD, int64_t nloc, int M1, int M2, double *dT,
                                    void *stream);
int dp_descriptor_contract_grad_f32(const float *T, const float *dD, int64_t nloc, int M1, int M2, float *dT,
                                    void *stream);

/* ------------------------------------------------------------------------
 * df64 variant: double inputs and outputs, double-float arithmetic.
 *
 * The same operations as the *_f64 calls above (Sec. II; same arguments,
 * layouts, limits, errors and nloc == 0 rule), computed in double-float
 * ("df64") arithmetic: every intermediate is the unevaluated sum of two
 * floats (48 significant bits), multiplied and accumulated through
 * error-free transformations on the FP32 pipes, which on GB300 retire 64
 * times the FP64 pipe's lanes per clock.  s, R~, dE/dT, dE/dD, T, D, ds and
 * dR~ are double arrays as in the *_f64 calls; results agree with them to a
 * few 1e-13 (max-norm relative on the paper's shapes; the rounding of df64
 * is 2^-48 per operation against 2^-53 in double).  Values must lie within
 * float's exponent range: magnitudes below ~1e-38 (relative parts below
 * ~1e-38 / 2^-24) flush towards zero, above ~3e38 overflow.
 *
 * dp_descriptor_contract_grad_df64 also stages dD_i: it needs
 * M1 (9 + M2) <= 7264 (DP_ERR_UNSUPPORTED beyond).
 *
 * The table is built for this arithmetic: [npair][nint][3][M1][4] float,
 * per interval the (a.hi, a.lo, b.hi, b.lo) vectors of all channels, then
 * (c, d), then (e, f) -- each coefficient of dp_table_build_f64 split into a
 * float and the float rounding of its remainder.
 * ---------------------------------------------------------------------- */
struct dp_env_info;
int dp_table_build_df64(const double *y, const double *dy, const double *d2y, int npair, int M1,
                        const dp_table_info *info, float *table, void *stream);
int dp_tabulate_fusion_fwd_moments_df64(const float *table, const dp_table_info *info, const double *s,
                                        const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                        int nnei, int ntypes, const int32_t *sel, int M1, double *T, void *stream);
int dp_tabulate_fusion_grad_moments_df64(const float *table, const dp_table_info *info, const double *s,
                                         const double *Rt, const int32_t *nvalid, const int32_t *atype, int64_t nloc,
                                         int nnei, int ntypes, const int32_t *sel, int M1, const double *dT,
                                         double *ds, double *dRt, void *stream);
int dp_descriptor_contract_df64(const double *T, int64_t nloc, int M1, int M2, double *D, void *stream);
int dp_descriptor_contract_grad_df64(const double *T, const double *dD, int64_t nloc, int M1, int M2, double *dT,
                                     void *stream);
/* dp_env_mat_f64 and dp_force_virial_f64 (declared below) in df64: the square root by Karp and
   Markstein's method, the reciprocal by a Newton-Raphson step, sin and cos of pi u by Taylor
   series on a reduced argument, each to about 2^-46 relative. */
int dp_env_mat_df64(const double *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes,
                    const int32_t *sel, const struct dp_env_info *env, double *s, double *Rt, int32_t *nvalid,
                    void *stream);
int dp_force_virial_df64(const double *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                         const struct dp_env_info *env, const double *ds, const double *dRt, double *F,
                         double *virial, void *stream);

/* ------------------------------------------------------------------------
 * Environment matrix front end and force / virial back end (Sec. II: the
 * weighting function s(r), the 4-vector rows and their normalisation; the
 * forces and virials follow from the derivatives of E with respect to atom i
 * and its neighbours).
 *
 * Coordinates: coord [nall][3], every position a neighbour list can point
 * at (local atoms first, nloc of them, then periodic images or ghost atoms,
 * as a domain decomposition provides them).  Neighbour list: nlist
 * [nloc][nnei] int32, row q of atom i holds the index j into coord of the
 * neighbour (the formatted list of Sec. II: per type segment the neighbours
 * sorted by distance, then -1 on every padding row).  d = coord[j] - coord[i].
 */
typedef struct dp_env_info {
  double rcs, rc;        /* smooth cutoff and cutoff, 0 < rcs < rc                     */
  int32_t kind;          /* 1: the paper's switch u^3(-6u^2+15u-10)+1; 0: cos(pi u)/2+1/2 */
  double mean, std;      /* normalisation of s: (s - mean) / std, std > 0 (0 and 1 = none) */
  double std_all;        /* normalisation of the xyz entries, > 0 (1 = none)           */
} dp_env_info;

/*
 * Rows of the environment matrix (Sec. II), u = (r - rcs)/(rc - rcs):
 *   s(r) = 1/r (r < rcs),  w(u)/r (rcs <= r < rc),  0 (r >= rc)
 *   R~ = ( (s(r) - mean)/std,  s(r) d_x/(r std_all),  s(r) d_y/(r std_all),  s(r) d_z/(r std_all) )
 * and s (the embedding input) = R~[0].  Rows with j < 0 are zero.
 *   coord [nall][3], nlist [nloc][nnei] inputs; env (host);
 *   s [nloc][nnei], Rt [nloc][nnei][4], nvalid [nloc][ntypes] int32 outputs
 *   (nvalid[i][b] = number of rows of segment b with j >= 0; with a formatted
 *   list these are the segment's first rows, as the fusion kernels expect).
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (nloc < 0, nnei < 1, sum(sel) != nnei),
 * DP_ERR_UNSUPPORTED (ntypes > DP_MAX_TYPES), DP_ERR_TABLE_INFO (env not as
 * stated), DP_ERR_CUDA.  nloc == 0 returns DP_OK without reading any pointer.
 * Indices j must lie in [0, nall); they are not checked on the device.
 */
int dp_env_mat_f64(const double *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes,
                   const int32_t *sel, const dp_env_info *env, double *s, double *Rt, int32_t *nvalid,
                   void *stream);
int dp_env_mat_f32(const float *coord, const int32_t *nlist, int64_t nloc, int nnei, int ntypes, const int32_t *sel,
                   const dp_env_info *env, float *s, float *Rt, int32_t *nvalid, void *stream);

/*
 * Forces and virial from ds = dE/ds [nloc][nnei] and dRt = dE/dR~
 * [nloc][nnei][4] (the outputs of dp_tabulate_fusion_grad_*), by the chain
 * rule through the rows above.  For a row (i, j) the gradient with respect to
 * d is
 *   g = (ds + dRt_0) s'(r)/(r std) d  +  (s'(r)/r^2 - s(r)/r^3) (dRt_xyz . d)/std_all d  +  s(r)/(r std_all) dRt_xyz
 * and F[i] += g, F[j] -= g (F = -dE/dr), virial[a][b] -= d_a g_b, summed
 * over all rows with j >= 0.
 *   F [nall][3] and virial [3][3] outputs, fully overwritten (forces on
 *   images / ghosts land on their own rows: fold them onto their owners as
 *   the domain decomposition requires).  Summation order is not fixed
 *   (atomic adds), so results agree with any serial order up to rounding.
 * Errors as dp_env_mat_* (nall < nloc is DP_ERR_SHAPE).
 */
int dp_force_virial_f64(const double *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                        const dp_env_info *env, const double *ds, const double *dRt, double *F, double *virial,
                        void *stream);
int dp_force_virial_f32(const float *coord, const int32_t *nlist, int64_t nloc, int64_t nall, int nnei,
                        const dp_env_info *env, const float *ds, const float *dRt, float *F, float *virial,
                        void *stream);

/* ------------------------------------------------------------------------
 * Fitting net (Sec. II: the descriptor D_i is passed to a fully connected
 * network that outputs the atomic energy E_i; the total energy is
 * E = sum_i E_i).  Each centre type t has its own net of nlayer layers with
 * widths widths[0..nlayer] (host), widths[0] = the length of D_i (M1 * M2),
 * widths[nlayer] = nout, the outputs per atom: 1 for the energy, M1 for the
 * weights a_i of the vector and tensor heads (dp_vector_head_*,
 * dp_tensor_head_*):
 *   v_0 = D_i
 *   v_l = tanh(v_{l-1} W_l + b_l) (+ v_{l-1} when widths[l] == widths[l-1]),  0 < l < nlayer
 *   E_i = v_{nlayer-1} W_nlayer + b_nlayer   (nout values)
 *   params      [ntypes][P]: per type, layer by layer, W_l [widths[l-1]][widths[l]]
 *               row-major then b_l [widths[l]]; P = sum_l (widths[l-1] + 1) widths[l].
 *   type_start  [ntypes + 1] HOST int64: the atoms of centre type t are rows
 *               type_start[t] .. type_start[t+1] - 1 (atoms sorted by centre
 *               type, as in every workload here); type_start[0] = 0 and
 *               nloc = type_start[ntypes].
 *   D    [nloc][widths[0]] input (the descriptor, flattened)
 *   E    [nloc][nout] output
 *   act  [nloc][H] output, H = the sum of the hidden widths: tanh(v_{l-1} W_l + b_l)
 *        of every hidden layer, in layer order -- what the backward needs.
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (a width outside [1, 2^20], type_start not
 * increasing or not starting at 0, more than 4,194,240 atoms of one type),
 * DP_ERR_UNSUPPORTED (nlayer or ntypes above DP_MAX_LAYERS / DP_MAX_TYPES),
 * DP_ERR_CUDA.  nloc == 0 reads no device pointer.
 */
int dp_fitting_fwd_f64(const double *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                       const double *D, double *E, double *act, void *stream);
int dp_fitting_fwd_f32(const float *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                       const float *D, float *E, float *act, void *stream);

/*
 * Backward of the fitting net: dD[i] = sum_c g_ic dE_ic/dD_i, the chain rule
 * through the layers in reverse (d tanh(z)/dz = 1 - tanh(z)^2; an identity
 * skip passes dE/dv_l on to v_{l-1}).
 *   act   [nloc][H] from dp_fitting_fwd_* on the same D
 *   g     [nloc][nout] upstream dE/dE_i, or NULL for all ones (nout = 1 only:
 *         E = sum_i E_i)
 *   dD    [nloc][widths[0]] output (feed it to dp_descriptor_contract_grad_*)
 *   work  [2][nloc][max hidden width] scratch, caller-owned, overwritten
 *         (NULL allowed when the net has a single hidden layer and nout = 1).
 * Errors as dp_fitting_fwd_*; a net without hidden layers is DP_ERR_UNSUPPORTED;
 * g NULL with nout > 1 is DP_ERR_NULL.
 */
int dp_fitting_grad_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                        const int64_t *type_start, const double *act, const double *g, double *dD, double *work,
                        void *stream);
int dp_fitting_grad_f32(const float *params, const int32_t *widths, int nlayer, int ntypes, const int64_t *type_start,
                        const float *act, const float *g, float *dD, float *work, void *stream);
/*
 * dp_fitting_grad_f64 without a work argument, for callers that cannot
 * allocate device memory or hand the library a scratch buffer -- an MD
 * engine that sizes all device memory at start-up and passes a plugin only
 * its inputs and outputs, where an allocation would synchronise the device
 * mid-step.  (The paper has no counterpart; this is an interface for such
 * callers.)  The scratch, 2 x nloc x (widest hidden layer) doubles, lives in
 * a fixed 8 MiB array inside the library (1,048,576 doubles: 2,184 atoms at
 * width 240), which every GPU that loads the library keeps until the process
 * exits; larger problems return DP_ERR_UNSUPPORTED -- use the call with a
 * work buffer.  Nothing is allocated: no cudaMalloc, no cudaFree, no
 * allocating library routine.  Every call looks the array's address up in
 * the current context (cudaGetSymbolAddress, which allocates nothing; the
 * first lookup on a device may load the library's kernels there, so make
 * the first call before any stream capture).  Every call on a device uses
 * the same array and it keeps the last call's contents; the kernels
 * overwrite every element they read, so nothing needs clearing, but calls
 * that overlap on the GPU (on
 * different streams, or from different threads) race on it.  Results are
 * those of dp_fitting_grad_f64.  Arguments and errors as dp_fitting_grad_f64.
 */
int dp_fitting_grad_noalloc_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                                const int64_t *type_start, const double *act, const double *g, double *dD,
                                void *stream);
/* The same in df64 arithmetic (double arrays; tanh itself in double). */
int dp_fitting_fwd_df64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                        const int64_t *type_start, const double *D, double *E, double *act, void *stream);
int dp_fitting_grad_df64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                         const int64_t *type_start, const double *act, const double *g, double *dD, double *work,
                         void *stream);

/*
 * The f64 fitting net with its hidden-layer GEMMs on the tensor cores
 * (tcgen05).  Same inputs, outputs and results as dp_fitting_fwd_f64 /
 * dp_fitting_grad_f64 (Sec. II: E_i from D_i, and dE_i/dD_i), to f64
 * accuracy: every GEMM operand element is split exactly into nine balanced
 * 6-bit digits scaled by its row's (A) or column's (B) power of two, the 45 digit
 * products that matter run as fp16 MMAs whose fp32 sums are exact integers
 * (at most 1792 of K per partial sum), and those sums are recombined exactly
 * before one rounding to f64.  Per output the error is below about
 * K 2^-49 max_k |a_ik| max_k |b_kj| (an f64 dot product: K 2^-53 sum_k
 * |a_ik b_kj|).  A row or column holding inf or NaN gives NaN outputs.  The
 * paper computes the net in double; this is that computation on hardware
 * whose FP64 rate is ~1000 times below its fp16 tensor rate.
 *   work, work_bytes  device scratch, caller-owned, 256-byte aligned, at least
 *                     dp_fitting_tc_work_bytes(widths, nlayer, nloc) bytes:
 *                     the operands' digit planes (the weights' rebuilt on
 *                     every call), partial results, and the [nloc][max hidden
 *                     width] buffers between layers.  Calls sharing a work
 *                     buffer must not overlap on the GPU.
 * One output: the output layer is a dot product per atom on the FP64 pipe.
 * Several outputs: the output layer (without tanh) and the backward's
 * g W_out^T are GEMMs on the tensor cores too.  Errors as the f64 calls, plus
 * DP_ERR_NULL / DP_ERR_SHAPE for a missing, short or misaligned work buffer.
 */
size_t dp_fitting_tc_work_bytes(const int32_t *widths, int nlayer, int64_t nloc); /* 0 on bad widths */
int dp_fitting_fwd_tc_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                          const int64_t *type_start, const double *D, double *E, double *act, void *work,
                          size_t work_bytes, void *stream);
int dp_fitting_grad_tc_f64(const double *params, const int32_t *widths, int nlayer, int ntypes,
                           const int64_t *type_start, const double *act, const double *g, double *dD, void *work,
                           size_t work_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Vector and tensor heads.  The paper's conclusion states that compression
 * carries over to DP models of vectors (dipoles) and tensors
 * (polarizabilities): their compressed path is the same up to T_i; the head
 * contracts the rotation-covariant rows k = 1..3 of T_i (the x, y, z columns
 * of R~, Sec. II) with M1 rotation-invariant weights a_i that a fitting net
 * with nout = M1 makes from D_i:
 *   vector:  v_i[c]    = sum_m a_i[m] T_i[1+c][m]
 *   tensor:  A_i[c][d] = sum_m a_i[m] (T_i[1+c][m] T_i[1+d][m])   (symmetric)
 * so v rotates as a vector and A as a rank-2 tensor when the coordinates do.
 *   T   [nloc][4][M1] input (dp_tabulate_fusion_fwd_*)
 *   a   [nloc][M1] input (dp_fitting_fwd_* with widths[nlayer] = M1)
 *   v   [nloc][3] output; A [nloc][3][3] output
 * Backward, from dE/dv [nloc][3] or dE/dA [nloc][3][3] (any, not only
 * symmetric):
 *   vector:  dT_i[1+c][m] = a_i[m] dv_i[c];  da_i[m] = sum_c dv_i[c] T_i[1+c][m]
 *   tensor:  dT_i[1+c][m] = a_i[m] sum_d (dA_i[c][d] + dA_i[d][c]) T_i[1+d][m];
 *            da_i[m] = sum_{c,d} dA_i[c][d] T_i[1+c][m] T_i[1+d][m]
 *   dT  [nloc][4][M1] output: overwritten (row k = 0 set to zero) when
 *       accumulate is 0; otherwise the head's dT is added to what dT holds
 *       (dE/dT of the descriptor, dp_descriptor_contract_grad_*), row 0 kept
 *   da  [nloc][M1] output (the upstream g of dp_fitting_grad_*)
 * Either output of the backward may be NULL (not computed), not both: a
 * model's backward takes da first (for the fitting net's backward, which
 * leads to the descriptor's dT) and then adds the head's dT to that.
 * All arrays device, row-major, caller-owned; nothing is allocated.
 * Errors: DP_ERR_NULL, DP_ERR_SHAPE (nloc < 0, M1 outside [1, 4096]),
 * DP_ERR_CUDA.  nloc == 0 reads no device pointer.
 */
int dp_vector_head_f64(const double *T, const double *a, int64_t nloc, int M1, double *v, void *stream);
int dp_vector_head_f32(const float *T, const float *a, int64_t nloc, int M1, float *v, void *stream);
int dp_vector_head_grad_f64(const double *T, const double *a, const double *dv, int64_t nloc, int M1, double *dT,
                            double *da, int accumulate, void *stream);
int dp_vector_head_grad_f32(const float *T, const float *a, const float *dv, int64_t nloc, int M1, float *dT,
                            float *da, int accumulate, void *stream);
int dp_tensor_head_f64(const double *T, const double *a, int64_t nloc, int M1, double *A, void *stream);
int dp_tensor_head_f32(const float *T, const float *a, int64_t nloc, int M1, float *A, void *stream);
int dp_tensor_head_grad_f64(const double *T, const double *a, const double *dA, int64_t nloc, int M1, double *dT,
                            double *da, int accumulate, void *stream);
int dp_tensor_head_grad_f32(const float *T, const float *a, const float *dA, int64_t nloc, int M1, float *dT,
                            float *da, int accumulate, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* DP_COMPRESS_H */
