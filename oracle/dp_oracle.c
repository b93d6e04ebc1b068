/*
 * Plain CPU oracle of the DP Compress tabulate-fusion path
 * (arXiv 2107.02103, Sec. II "Methods"; supplementary material).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load or call this file.  It shares no
 * code, header, table, constant or helper with the CUDA library and never
 * calls it; the two only meet through the seeded inputs of `workloads`.
 *
 * Everything is written as the paper states it, in the paper's order and
 * notation, with no blocking, fusion or reordering:
 *   - the embedding net G_m(s) and its first two derivatives (Sec. II, the
 *     embedding matrix; the tanh activation and residual skips are the
 *     embedding-net structure the workloads specify), in long double;
 *   - the table nodes x_l and the six-coefficient quintic per interval and
 *     channel from (y, y', y'') at both ends (Sec. II, the constraint
 *     equations and the closed forms for a..f), in long double, rounded once;
 *   - the interval search and the local variable t = x - x_l;
 *   - the forward contraction T_i = (1/N_c) R~_i^T G_i with G evaluated from
 *     the table only for valid neighbours (Sec. II, kernel fusion and the
 *     skip of padded rows), in double;
 *   - its gradient dE/ds and dE/dR~ from an upstream dE/dT, in double;
 *   - the descriptor D_i = S_i (S_i^<)^T with S_i = T_i^T (Sec. II), and its
 *     gradient dE/dT from an upstream dE/dD, in double;
 *   - the embedding matrix G itself, through the table or straight from the
 *     net, for the explicit and uncompressed comparisons;
 *   - the environment matrix from coordinates and a neighbour list (Sec. II,
 *     the weighting function s(r) and the 4-vector rows with their
 *     normalisation), and the forces and virial that follow from dE/ds and
 *     dE/dR~ by the chain rule through those rows.
 *
 * Pins: every function here is pinned by tests that do not re-run its own
 * formula (closed forms, exactly reproduced polynomials, a sin() error
 * bound, finite differences, symmetries, brute force, mutations).  No
 * function is "parity unpinned".
 *
 * Build: gcc -O2 -ffp-contract=off [-fopenmp] -shared -fPIC.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

typedef long double ld;

/* Table range: fine segment [lower, upper) with step stride0 (n0 intervals),
   coarse segment [upper, upper_ext) with step stride1 (n1 intervals). */
typedef struct {
  double lower, upper, upper_ext, stride0, stride1;
  int32_t n0, n1;
} or_info;

#define OR_MAXW 1024

/* ------------------------------------------------------- embedding net */

/*
 * Embedding net G(x): widths[0] = 1 input, widths[nlayer] = M outputs.
 * Layer l maps v (width a) to u (width b) with z = v W_l + b_l, h = tanh(z),
 *   u = h + v        when b == a,
 *   u = h + (v, v)   when b == 2a,
 *   u = h            otherwise.
 * params holds, layer by layer, W_l [a][b] row-major then b_l [b].
 * The first and second derivatives in x are carried in forward mode:
 *   z' = v' W, z'' = v'' W, h' = (1 - h^2) z', h'' = (1 - h^2) z'' - 2 h (1 - h^2) z'^2.
 * Returns 0, or -1 for a width above OR_MAXW.
 */
int or_net_eval(const double *params, const int32_t *widths, int nlayer, double x, double *y, double *dy,
                double *d2y) {
  ld v[OR_MAXW], v1[OR_MAXW], v2[OR_MAXW], u[OR_MAXW], u1[OR_MAXW], u2[OR_MAXW];
  for (int l = 0; l <= nlayer; ++l)
    if (widths[l] < 1 || widths[l] > OR_MAXW) return -1;
  if (widths[0] != 1) return -1;
  v[0] = (ld)x;
  v1[0] = 1.0L;
  v2[0] = 0.0L;
  const double *p = params;
  for (int l = 0; l < nlayer; ++l) {
    int a = widths[l], b = widths[l + 1];
    const double *W = p, *bias = p + (size_t)a * b;
    p += (size_t)a * b + b;
    for (int o = 0; o < b; ++o) {
      ld z = (ld)bias[o], z1 = 0.0L, z2 = 0.0L;
      for (int i = 0; i < a; ++i) {
        ld w = (ld)W[(size_t)i * b + o];
        z += v[i] * w;
        z1 += v1[i] * w;
        z2 += v2[i] * w;
      }
      ld h = tanhl(z);
      ld sech2 = 1.0L - h * h;
      ld h1 = sech2 * z1;
      ld h2 = sech2 * z2 - 2.0L * h * sech2 * z1 * z1;
      if (b == a) {
        u[o] = h + v[o];
        u1[o] = h1 + v1[o];
        u2[o] = h2 + v2[o];
      } else if (b == 2 * a) {
        u[o] = h + v[o % a];
        u1[o] = h1 + v1[o % a];
        u2[o] = h2 + v2[o % a];
      } else {
        u[o] = h;
        u1[o] = h1;
        u2[o] = h2;
      }
    }
    for (int o = 0; o < b; ++o) {
      v[o] = u[o];
      v1[o] = u1[o];
      v2[o] = u2[o];
    }
  }
  int M = widths[nlayer];
  for (int m = 0; m < M; ++m) {
    if (y) y[m] = (double)v[m];
    if (dy) dy[m] = (double)v1[m];
    if (d2y) d2y[m] = (double)v2[m];
  }
  return 0;
}

/*
 * G and G' at a list of inputs: xs[n] with pair[n] choosing the parameter row
 * (params is [npair][P]).  G, dG are [n][M]; dG may be NULL.
 */
int or_net_rows(const double *params, int64_t P, const int32_t *widths, int nlayer, const double *xs,
                const int32_t *pair, int64_t n, double *G, double *dG, int nthreads) {
  int M = widths[nlayer];
  int err = 0;
#ifdef _OPENMP
  if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 16) reduction(| : err)
#endif
  for (int64_t q = 0; q < n; ++q) {
    const double *pp = params + (size_t)pair[q] * P;
    if (or_net_eval(pp, widths, nlayer, xs[q], G + (size_t)q * M, dG ? dG + (size_t)q * M : NULL, NULL)) err |= 1;
  }
  return err ? -1 : 0;
}

/* ---------------------------------------------------------- table range */

/*
 * Table range from a scan of the data (Sec. II: the interpolated range is
 * set from the training data, and its upper bound covers the largest value
 * found there), extended by a coarse segment up to ext * upper:
 *   lower = 0 when every s >= 0, else stride0 * floor(s_min / stride0)
 *   upper = stride1 * ceil(s_max / stride1)
 *   upper_ext = ext * upper
 *   n0 = (upper - lower) / stride0, n1 = (upper_ext - upper) / stride1 (rounded).
 * Returns -1 when the range is empty or the steps are not positive.
 */
int or_table_info(double s_min, double s_max, double stride0, double stride1, double ext, or_info *out) {
  if (!(stride0 > 0.0) || !(stride1 > 0.0) || !(ext >= 1.0) || !(s_max > 0.0) || !(s_min <= s_max)) return -1;
  out->lower = s_min >= 0.0 ? 0.0 : stride0 * floor(s_min / stride0);
  out->upper = stride1 * ceil(s_max / stride1);
  out->upper_ext = ext * out->upper;
  out->stride0 = stride0;
  out->stride1 = stride1;
  out->n0 = (int32_t)llround((out->upper - out->lower) / stride0);
  out->n1 = (int32_t)llround((out->upper_ext - out->upper) / stride1);
  if (out->n0 < 1) return -1;
  return 0;
}

/* node x_l, l = 0 .. n0 + n1 (Sec. II: x_1 .. x_{L+1}, here 0-based) */
double or_node_x(const or_info *in, int32_t l) {
  if (l < in->n0) return in->lower + (double)l * in->stride0;
  if (l == in->n0) return in->upper;
  return in->upper + (double)(l - in->n0) * in->stride1;
}

/* y, y', y'' of every channel at every node: [nint + 1][M] each */
int or_nodes(const double *params, const int32_t *widths, int nlayer, const or_info *in, double *y, double *dy,
             double *d2y) {
  int M = widths[nlayer];
  int32_t nn = in->n0 + in->n1 + 1;
  for (int32_t l = 0; l < nn; ++l) {
    int r = or_net_eval(params, widths, nlayer, or_node_x(in, l), y + (size_t)l * M, dy + (size_t)l * M,
                        d2y + (size_t)l * M);
    if (r) return r;
  }
  return 0;
}

/* ---------------------------------------------------------- table build */

/*
 * Coefficients of g_m^l(t) = a t^5 + b t^4 + c t^3 + d t^2 + e t + f on
 * interval l, t = x - x_l in [0, Dt), from y, y', y'' at x_l and x_{l+1}
 * (Sec. II, the closed forms for a..f with h = y_{l+1} - y_l and
 * Dt = x_{l+1} - x_l):
 *   a = [12h - 6(y'_{l+1} + y'_l)Dt + (y''_{l+1} - y''_l)Dt^2] / (2 Dt^5)
 *   b = [-30h + (14y'_{l+1} + 16y'_l)Dt + (3y''_l - 2y''_{l+1})Dt^2] / (2 Dt^4)
 *   c = [20h - (8y'_{l+1} + 12y'_l)Dt - (3y''_l - y''_{l+1})Dt^2] / (2 Dt^3)
 *   d = y''_l / 2,  e = y'_l,  f = y_l.
 * The local variable t (not the absolute x) is the reading under which these
 * forms match y, y', y'' at both ends.  Dt is stride0 on the fine segment and
 * stride1 on the coarse one.  Computed in long double, rounded once.
 * y, dy, d2y: [nint + 1][M]; table: [nint][M][6] = (a, b, c, d, e, f).
 */
void or_table_build(const double *y, const double *dy, const double *d2y, int M, const or_info *in,
                    double *table) {
  int32_t nint = in->n0 + in->n1;
  for (int32_t l = 0; l < nint; ++l) {
    ld Dt = (ld)(l < in->n0 ? in->stride0 : in->stride1);
    ld Dt2 = Dt * Dt, Dt3 = Dt2 * Dt, Dt4 = Dt3 * Dt, Dt5 = Dt4 * Dt;
    for (int m = 0; m < M; ++m) {
      ld y0 = y[(size_t)l * M + m], y1 = y[(size_t)(l + 1) * M + m];
      ld p0 = dy[(size_t)l * M + m], p1 = dy[(size_t)(l + 1) * M + m];
      ld q0 = d2y[(size_t)l * M + m], q1 = d2y[(size_t)(l + 1) * M + m];
      ld h = y1 - y0;
      ld a = (12.0L * h - 6.0L * (p1 + p0) * Dt + (q1 - q0) * Dt2) / (2.0L * Dt5);
      ld b = (-30.0L * h + (14.0L * p1 + 16.0L * p0) * Dt + (3.0L * q0 - 2.0L * q1) * Dt2) / (2.0L * Dt4);
      ld c = (20.0L * h - (8.0L * p1 + 12.0L * p0) * Dt - (3.0L * q0 - q1) * Dt2) / (2.0L * Dt3);
      double *out = table + ((size_t)l * M + m) * 6;
      out[0] = (double)a;
      out[1] = (double)b;
      out[2] = (double)c;
      out[3] = (double)(q0 / 2.0L);
      out[4] = (double)p0;
      out[5] = (double)y0;
    }
  }
}

/*
 * Derivative `order` (0, 1, 2) of interval l's polynomial at local t, all M
 * channels, evaluated in long double from the stored double coefficients.
 */
void or_poly_eval(const double *table, int M, int32_t l, double t, int order, double *out) {
  ld T = (ld)t;
  for (int m = 0; m < M; ++m) {
    const double *c = table + ((size_t)l * M + m) * 6;
    ld a = c[0], b = c[1], cc = c[2], d = c[3], e = c[4], f = c[5];
    ld v;
    if (order == 0)
      v = a * T * T * T * T * T + b * T * T * T * T + cc * T * T * T + d * T * T + e * T + f;
    else if (order == 1)
      v = 5.0L * a * T * T * T * T + 4.0L * b * T * T * T + 3.0L * cc * T * T + 2.0L * d * T + e;
    else
      v = 20.0L * a * T * T * T + 12.0L * b * T * T + 6.0L * cc * T + 2.0L * d;
    out[m] = (double)v;
  }
}

/* ------------------------------------------------------ interval search */

/*
 * Interval l and local variable t = x - x_l for input x.
 *   lower <= x < upper:      l = floor((x - lower) / stride0), kept in [0, n0 - 1]
 *   upper <= x < upper_ext:  l = n0 + floor((x - upper) / stride1), kept in [n0, n0 + n1 - 1]
 *   x < lower:               l = 0, t = 0 (the first node), returns 1
 *   x >= upper_ext:          l = last, t = its width (the last node), returns 1
 *   x NaN:                   l = 0, t = NaN, returns 0 (NaN reaches the results)
 * A return of 1 marks a clamped input: the tabulated function is extended by
 * its end value there, so its derivative is 0.
 */
int or_locate(const or_info *in, double x, int32_t *l, double *t) {
  int32_t nint = in->n0 + in->n1;
  if (isnan(x)) {
    *l = 0;
    *t = x;
    return 0;
  }
  if (x < in->lower) {
    *l = 0;
    *t = 0.0;
    return 1;
  }
  if (x >= in->upper_ext || (x >= in->upper && in->n1 == 0)) {
    *l = nint - 1;
    *t = (in->n1 > 0) ? in->stride1 : in->stride0;
    return 1;
  }
  int32_t k;
  if (x < in->upper) {
    k = (int32_t)floor((x - in->lower) / in->stride0);
    if (k < 0) k = 0;
    if (k > in->n0 - 1) k = in->n0 - 1;
  } else {
    k = in->n0 + (int32_t)floor((x - in->upper) / in->stride1);
    if (k < in->n0) k = in->n0;
    if (k > nint - 1) k = nint - 1;
  }
  *l = k;
  *t = x - or_node_x(in, k);
  return 0;
}

/* g(t) = a t^5 + b t^4 + c t^3 + d t^2 + e t + f and g'(t) (Sec. II) */
static double poly_g(const double *c, double t) {
  double t2 = t * t, t3 = t2 * t, t4 = t3 * t, t5 = t4 * t;
  return c[0] * t5 + c[1] * t4 + c[2] * t3 + c[3] * t2 + c[4] * t + c[5];
}
static double poly_dg(const double *c, double t) {
  double t2 = t * t, t3 = t2 * t, t4 = t3 * t;
  return 5.0 * c[0] * t4 + 4.0 * c[1] * t3 + 3.0 * c[2] * t2 + 2.0 * c[3] * t + c[4];
}

/* ------------------------------------------------- forward contraction */

static int check_counts(const int32_t *nvalid, int64_t i, int ntypes, const int32_t *sel) {
  for (int b = 0; b < ntypes; ++b) {
    int32_t nv = nvalid[i * ntypes + b];
    if (nv < 0 || nv > sel[b]) return 1;
  }
  return 0;
}

/*
 * T_i = (1/N_c) R~_i^T G_i, 4 x M per atom, with row j of G_i evaluated from
 * the table only for valid neighbours (Sec. II: the column of G_i^T is formed
 * and multiplied into R~ only when j is a valid neighbour; rows after the
 * last real neighbour of a type segment are zero and are skipped).
 *   T[a][k][m] = (1/N_c) sum_{beta} sum_{j < nvalid[i][beta]} R~[i][o_beta + j][k] g_m(s[i][o_beta + j])
 * with i = atoms[a] (or a when atoms is NULL), o_beta = sum of sel before
 * beta, N_c = nnei = sum of sel, and the table of pair (atype[i], beta).
 * table: [npair][nint][M][6].  Returns -1 on a count outside [0, sel].
 */
int or_fwd(const double *table, const or_info *in, const double *s, const double *Rt, const int32_t *nvalid,
           const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M, const int64_t *atoms,
           int64_t natoms, double *T, int nthreads) {
  int32_t nint = in->n0 + in->n1;
  int off[64];
  int acc = 0;
  for (int b = 0; b < ntypes; ++b) {
    off[b] = acc;
    acc += sel[b];
  }
  int err = 0;
  (void)nloc;
#ifdef _OPENMP
  if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 4) reduction(| : err)
#endif
  for (int64_t a = 0; a < natoms; ++a) {
    int64_t i = atoms ? atoms[a] : a;
    double *Ti = T + (size_t)a * 4 * M;
    for (int q = 0; q < 4 * M; ++q) Ti[q] = 0.0;
    if (check_counts(nvalid, i, ntypes, sel)) {
      err |= 1;
      continue;
    }
    int alpha = atype ? atype[i] : 0;
    for (int beta = 0; beta < ntypes; ++beta) {
      const double *tab = table + (size_t)(alpha * ntypes + beta) * nint * M * 6;
      for (int j = 0; j < nvalid[i * ntypes + beta]; ++j) {
        int64_t row = i * nnei + off[beta] + j;
        int32_t l;
        double t;
        or_locate(in, s[row], &l, &t);
        for (int m = 0; m < M; ++m) {
          double g = poly_g(tab + ((size_t)l * M + m) * 6, t);
          for (int k = 0; k < 4; ++k) Ti[k * M + m] += Rt[row * 4 + k] * g;
        }
      }
    }
    for (int q = 0; q < 4 * M; ++q) Ti[q] = Ti[q] / (double)nnei;
  }
  return err ? -1 : 0;
}

/*
 * Gradient of E through T_i given the upstream dT = dE/dT_i (4 x M per atom):
 *   dE/dR~[i][row][k] = (1/N_c) sum_m dT[k][m] g_m(s_row)
 *   dE/ds[i][row]     = (1/N_c) sum_m (sum_k dT[k][m] R~[i][row][k]) g'_m(s_row)
 * for valid rows; g' = 0 where the interval search clamped s; padded rows
 * get 0 (they are constants, not functions of the coordinates).
 * ds: [natoms][nnei], dRt: [natoms][nnei][4], indexed like T in or_fwd;
 * dT: [nloc][4][M] indexed by i.
 */
int or_grad(const double *table, const or_info *in, const double *s, const double *Rt, const int32_t *nvalid,
            const int32_t *atype, int64_t nloc, int nnei, int ntypes, const int32_t *sel, int M, const double *dT,
            const int64_t *atoms, int64_t natoms, double *ds, double *dRt, int nthreads) {
  int32_t nint = in->n0 + in->n1;
  int off[64];
  int acc = 0;
  for (int b = 0; b < ntypes; ++b) {
    off[b] = acc;
    acc += sel[b];
  }
  int err = 0;
  (void)nloc;
#ifdef _OPENMP
  if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 4) reduction(| : err)
#endif
  for (int64_t a = 0; a < natoms; ++a) {
    int64_t i = atoms ? atoms[a] : a;
    double *dsa = ds + (size_t)a * nnei;
    double *dRa = dRt + (size_t)a * nnei * 4;
    for (int q = 0; q < nnei; ++q) dsa[q] = 0.0;
    for (int q = 0; q < 4 * nnei; ++q) dRa[q] = 0.0;
    if (check_counts(nvalid, i, ntypes, sel)) {
      err |= 1;
      continue;
    }
    const double *dTi = dT + (size_t)i * 4 * M;
    int alpha = atype ? atype[i] : 0;
    for (int beta = 0; beta < ntypes; ++beta) {
      const double *tab = table + (size_t)(alpha * ntypes + beta) * nint * M * 6;
      for (int j = 0; j < nvalid[i * ntypes + beta]; ++j) {
        int r = off[beta] + j;
        int64_t row = i * nnei + r;
        int32_t l;
        double t;
        int clamped = or_locate(in, s[row], &l, &t);
        double dsum = 0.0, dr[4] = {0.0, 0.0, 0.0, 0.0};
        for (int m = 0; m < M; ++m) {
          const double *c = tab + ((size_t)l * M + m) * 6;
          double g = poly_g(c, t);
          double dg = clamped ? 0.0 : poly_dg(c, t);
          double rm = 0.0;
          for (int k = 0; k < 4; ++k) rm += dTi[k * M + m] * Rt[row * 4 + k];
          dsum += rm * dg;
          for (int k = 0; k < 4; ++k) dr[k] += dTi[k * M + m] * g;
        }
        dsa[r] = dsum / (double)nnei;
        for (int k = 0; k < 4; ++k) dRa[(size_t)r * 4 + k] = dr[k] / (double)nnei;
      }
    }
  }
  return err ? -1 : 0;
}

/*
 * Descriptor (Sec. II): S_i = T_i^T is M x 4, S_i^< its first M2 rows,
 * D_i = S_i (S_i^<)^T is M x M2:  D[a][m][n] = sum_k T[a][k][m] T[a][k][n].
 */
void or_descriptor(const double *T, int64_t n, int M, int M2, double *D) {
  for (int64_t a = 0; a < n; ++a) {
    const double *Ta = T + (size_t)a * 4 * M;
    double *Da = D + (size_t)a * M * M2;
    for (int m = 0; m < M; ++m)
      for (int q = 0; q < M2; ++q) {
        double v = 0.0;
        for (int k = 0; k < 4; ++k) v += Ta[k * M + m] * Ta[k * M + q];
        Da[(size_t)m * M2 + q] = v;
      }
  }
}

/*
 * Gradient of the descriptor.  D[m][n] = sum_k T[k][m] T[k][n] (n < M2) is
 * quadratic in T, so for an upstream dD = dE/dD ([n][M][M2] like D):
 *   dE/dT[k][m] = sum_{n<M2} dD[m][n] T[k][n]  +  [m < M2] sum_{m'} dD[m'][m] T[k][m']
 * (the first term through the S_i factor, the second through S_i^<).
 */
void or_descriptor_grad(const double *T, const double *dD, int64_t n, int M, int M2, double *dT) {
  for (int64_t a = 0; a < n; ++a) {
    const double *Ta = T + (size_t)a * 4 * M;
    const double *Ga = dD + (size_t)a * M * M2;
    double *dTa = dT + (size_t)a * 4 * M;
    for (int k = 0; k < 4; ++k)
      for (int m = 0; m < M; ++m) {
        double v = 0.0;
        for (int q = 0; q < M2; ++q) v += Ga[(size_t)m * M2 + q] * Ta[k * M + q];
        if (m < M2)
          for (int mp = 0; mp < M; ++mp) v += Ga[(size_t)mp * M2 + m] * Ta[k * M + mp];
        dTa[k * M + m] = v;
      }
  }
}

/*
 * The embedding matrix itself, through the table, for EVERY row (valid and
 * padding alike, no skip): G[a][row][m] = g_m(s[i][row]) with the table of
 * pair (atype[i], type of row).  The original workflow forms this matrix and
 * multiplies it into R~ with a GEMM (Sec. II, Fig. 1(b)); tests do that
 * product with a library matmul and compare with or_fwd.
 */
void or_embed_rows(const double *table, const or_info *in, const double *s, const int32_t *atype, int nnei,
                   int ntypes, const int32_t *sel, int M, const int64_t *atoms, int64_t natoms, double *G,
                   double *dG) {
  int32_t nint = in->n0 + in->n1;
  for (int64_t a = 0; a < natoms; ++a) {
    int64_t i = atoms ? atoms[a] : a;
    int alpha = atype ? atype[i] : 0;
    int r = 0;
    for (int beta = 0; beta < ntypes; ++beta)
      for (int j = 0; j < sel[beta]; ++j, ++r) {
        const double *tab = table + (size_t)(alpha * ntypes + beta) * nint * M * 6;
        int32_t l;
        double t;
        int clamped = or_locate(in, s[i * nnei + r], &l, &t);
        for (int m = 0; m < M; ++m) {
          const double *c = tab + ((size_t)l * M + m) * 6;
          G[((size_t)a * nnei + r) * M + m] = poly_g(c, t);
          if (dG) dG[((size_t)a * nnei + r) * M + m] = clamped ? 0.0 : poly_dg(c, t);
        }
      }
  }
}

/* ------------------------------------------------- environment matrix */

/*
 * Weighting function s(r) and its derivative (Sec. II).  With
 * u = (r - rcs)/(rc - rcs):
 *   r < rcs:         s = 1/r
 *   rcs <= r < rc:   s = w(u)/r
 *   r >= rc:         s = 0
 * kind 1 is the paper's switch w = u^3 (-6u^2 + 15u - 10) + 1; kind 0 is the
 * cosine switch of the benchmark configurations, w = cos(pi u)/2 + 1/2.
 */
static void or_weight(double r, double rcs, double rc, int kind, double *sv, double *dsv) {
  if (r < rcs) {
    *sv = 1.0 / r;
    *dsv = -1.0 / (r * r);
    return;
  }
  if (r >= rc) {
    *sv = 0.0;
    *dsv = 0.0;
    return;
  }
  double u = (r - rcs) / (rc - rcs);
  double w, dw;  /* w(u) and dw/du */
  if (kind == 1) {
    w = u * u * u * (-6.0 * u * u + 15.0 * u - 10.0) + 1.0;
    dw = -30.0 * u * u * (u - 1.0) * (u - 1.0);
  } else {
    const double pi = 3.14159265358979323846;
    w = 0.5 * cos(pi * u) + 0.5;
    dw = -0.5 * pi * sin(pi * u);
  }
  *sv = w / r;
  *dsv = dw / ((rc - rcs) * r) - w / (r * r);
}

double or_switch(double r, double rcs, double rc, int kind, double *ds_dr) {
  double sv, dsv;
  or_weight(r, rcs, rc, kind, &sv, &dsv);
  if (ds_dr) *ds_dr = dsv;
  return sv;
}

/*
 * Rows of the environment matrix (Sec. II).  For atom i < nloc and row q of
 * nlist (index j into coord, -1 on padding rows): d = r_j - r_i, r = |d|,
 *   R~ = ( (s(r) - mean)/std,  s(r) d_x / r / std_all,  s(r) d_y / r / std_all,  s(r) d_z / r / std_all )
 * with norm = {mean, std, std_all} (NULL: {0, 1, 1}); the embedding input
 * s of the row is its first entry.  Padding rows are zero.
 */
void or_env_mat(int64_t nloc, const double *coord, const int32_t *nlist, int nnei, double rcs, double rc, int kind,
                const double *norm, double *s, double *Rt) {
  const double mean = norm ? norm[0] : 0.0, sd = norm ? norm[1] : 1.0, sa = norm ? norm[2] : 1.0;
  for (int64_t i = 0; i < nloc; ++i)
    for (int q = 0; q < nnei; ++q) {
      const int64_t row = i * nnei + q;
      const int32_t j = nlist[row];
      if (j < 0) {
        s[row] = 0.0;
        for (int k = 0; k < 4; ++k) Rt[4 * row + k] = 0.0;
        continue;
      }
      double d[3], r2 = 0.0;
      for (int a = 0; a < 3; ++a) {
        d[a] = coord[3 * (int64_t)j + a] - coord[3 * i + a];
        r2 += d[a] * d[a];
      }
      const double r = sqrt(r2);
      const double sv = or_switch(r, rcs, rc, kind, NULL);
      const double sh = (sv - mean) / sd;
      s[row] = sh;
      Rt[4 * row + 0] = sh;
      for (int a = 0; a < 3; ++a) Rt[4 * row + 1 + a] = sv * d[a] / r / sa;
    }
}

/*
 * Forces and virial from the gradients of the rows (the derivatives of E_i
 * with respect to atom i and its neighbours, Sec. II).  For a valid row
 * (i, j) with d = r_j - r_i, the energy depends on d through s (the
 * embedding input) and R~; with ds = dE/ds and dR = dE/dR~ of the row,
 *   dE/dd_b = (ds + dR_0) s'(r) d_b / (r std)
 *           + sum_a dR_{1+a} / std_all * ( s'(r) d_a d_b / r^2 + s(r) (delta_ab / r - d_a d_b / r^3) ).
 * Then F_i += dE/dd, F_j -= dE/dd (F = -dE/dr; d = r_j - r_i), and the
 * virial W_ab = - sum over rows of d_a dE/dd_b.  F has nall rows (every
 * index nlist can hold); both outputs are overwritten.
 */
void or_force_virial(int64_t nloc, int64_t nall, const double *coord, const int32_t *nlist, int nnei, double rcs,
                     double rc, int kind, const double *norm, const double *ds, const double *dRt, double *F,
                     double *W) {
  const double sd = norm ? norm[1] : 1.0, sa = norm ? norm[2] : 1.0;
  for (int64_t a = 0; a < 3 * nall; ++a) F[a] = 0.0;
  for (int a = 0; a < 9; ++a) W[a] = 0.0;
  for (int64_t i = 0; i < nloc; ++i)
    for (int q = 0; q < nnei; ++q) {
      const int64_t row = i * nnei + q;
      const int32_t j = nlist[row];
      if (j < 0) continue;
      double d[3], r2 = 0.0;
      for (int a = 0; a < 3; ++a) {
        d[a] = coord[3 * (int64_t)j + a] - coord[3 * i + a];
        r2 += d[a] * d[a];
      }
      const double r = sqrt(r2);
      double sv, dsv;
      or_weight(r, rcs, rc, kind, &sv, &dsv);
      double g[3];
      for (int b = 0; b < 3; ++b) {
        double v = (ds[row] + dRt[4 * row + 0]) * dsv * d[b] / (r * sd);
        for (int a = 0; a < 3; ++a) {
          const double dab = (a == b) ? 1.0 : 0.0;
          v += dRt[4 * row + 1 + a] / sa * (dsv * d[a] * d[b] / r2 + sv * (dab / r - d[a] * d[b] / (r2 * r)));
        }
        g[b] = v;
      }
      for (int b = 0; b < 3; ++b) {
        F[3 * i + b] += g[b];
        F[3 * (int64_t)j + b] -= g[b];
      }
      for (int a = 0; a < 3; ++a)
        for (int b = 0; b < 3; ++b) W[3 * a + b] -= d[a] * g[b];
    }
}

/* ----------------------------------------------------------- fitting net */

/*
 * Fitting net (Sec. II: the descriptor D_i is passed to a fully connected
 * network that outputs the atomic energy E_i; the total energy is
 * E = sum_i E_i).  For centre type t the net has nlayer layers with widths
 * widths[0..nlayer], widths[0] = the length of D_i, widths[nlayer] = nout
 * (1 for the energy; M1 for the vector and tensor heads below, the models the
 * conclusion of the paper says compression carries over to):
 *   hidden layer l (l < nlayer - 1):  v_l = tanh(v_{l-1} W_l + b_l) (+ v_{l-1} when the widths agree)
 *   output layer:                     E_i = v_{nlayer-1} W_nlayer + b_nlayer   (nout values)
 * params [ntypes][P], layer by layer W_l [a][b] row-major then b_l [b].
 * E [n][nout]; when dD is not NULL also sum_c g[i][c] dE_ic/dD_i [n][widths[0]]
 * by the chain rule backwards through the layers (d tanh(z)/dz = 1 - tanh(z)^2),
 * g [n][nout] (NULL: all 1).  Returns -1 for a width above OR_FITW or bad sizes.
 */
#define OR_FITW 4096
int or_fitting(const double *params, int64_t P, const int32_t *widths, int nlayer, const double *D,
               const int32_t *atype, int64_t n, const double *g, double *E, double *dD, int nthreads) {
  if (nlayer < 1) return -1;
  const int nout = widths[nlayer];
  int hid = 0;  // sum of the hidden widths
  for (int l = 0; l <= nlayer; ++l)
    if (widths[l] < 1 || widths[l] > OR_FITW) return -1;
  for (int l = 1; l < nlayer; ++l) hid += widths[l];
  int err = 0;
#ifdef _OPENMP
  if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 4) reduction(| : err)
#endif
  for (int64_t i = 0; i < n; ++i) {
    double *act = malloc(sizeof(double) * (size_t)(hid + widths[0]));  // the layer outputs v_0 .. v_{nlayer-1}
    double *tn = malloc(sizeof(double) * (size_t)(hid > 0 ? hid : 1));  // tanh of every hidden layer
    double *gv = malloc(sizeof(double) * (size_t)OR_FITW * 2);
    if (!act || !tn || !gv) {
      err |= 1;
      free(act);
      free(tn);
      free(gv);
      continue;
    }
    const double *pp = params + (size_t)(atype ? atype[i] : 0) * P;
    for (int k = 0; k < widths[0]; ++k) act[k] = D[(size_t)i * widths[0] + k];
    // forward
    const double *p = pp;
    int off_in = 0, off_out = widths[0], off_t = 0;
    for (int l = 1; l < nlayer; ++l) {
      const int a = widths[l - 1], b = widths[l];
      const double *W = p, *bias = p + (size_t)a * b;
      p += (size_t)a * b + b;
      for (int o = 0; o < b; ++o) {
        double z = bias[o];
        for (int k = 0; k < a; ++k) z += act[off_in + k] * W[(size_t)k * b + o];
        const double t = tanh(z);
        tn[off_t + o] = t;
        act[off_out + o] = t + (b == a ? act[off_in + o] : 0.0);
      }
      off_in = off_out;
      off_out += b;
      off_t += b;
    }
    const int a = widths[nlayer - 1];
    const double *Wo = p, *bo = p + (size_t)a * nout;
    for (int c = 0; c < nout; ++c) {
      double e = bo[c];
      for (int k = 0; k < a; ++k) e += act[off_in + k] * Wo[(size_t)k * nout + c];
      E[(size_t)i * nout + c] = e;
    }
    if (dD) {
      // backward: gv holds dE_i/dv_l for the current layer (E_i weighted by g)
      double *cur = gv, *nxt = gv + OR_FITW;
      for (int k = 0; k < a; ++k) {
        double v = 0.0;
        for (int c = 0; c < nout; ++c) v += (g ? g[(size_t)i * nout + c] : 1.0) * Wo[(size_t)k * nout + c];
        cur[k] = v;
      }
      // walk the hidden layers from the last to the first; their parameters precede Wo
      const double *pl = Wo;
      int toff = off_t;
      for (int l = nlayer - 1; l >= 1; --l) {
        const int ai = widths[l - 1], bo_ = widths[l];
        pl -= (size_t)ai * bo_ + bo_;
        const double *W = pl;
        toff -= bo_;
        for (int k = 0; k < ai; ++k) nxt[k] = 0.0;
        for (int o = 0; o < bo_; ++o) {
          const double t = tn[toff + o];
          const double gz = cur[o] * (1.0 - t * t);
          for (int k = 0; k < ai; ++k) nxt[k] += gz * W[(size_t)k * bo_ + o];
        }
        if (bo_ == ai)
          for (int k = 0; k < ai; ++k) nxt[k] += cur[k];
        double *s = cur;
        cur = nxt;
        nxt = s;
      }
      for (int k = 0; k < widths[0]; ++k) dD[(size_t)i * widths[0] + k] = cur[k];
    }
    free(act);
    free(tn);
    free(gv);
  }
  return err ? -1 : 0;
}

/* --------------------------------------------- vector and tensor heads */

/*
 * Vector and tensor DP models (the paper's conclusion: compression carries
 * over to models of vectors, such as dipoles, and of tensors, such as
 * polarizabilities).  The compressed path is the same up to T_i; the head
 * contracts the rotation-covariant rows k = 1..3 of T_i (the x, y, z columns
 * of R~, Sec. II) with the fitting net's M outputs a_i, which are invariant:
 *   vector:  v_i[c]    = sum_m a_i[m] T_i[1+c][m]
 *   tensor:  A_i[c][d] = sum_m a_i[m] (T_i[1+c][m] T_i[1+d][m])   (symmetric to the bit)
 * T [n][4][M], a [n][M], v [n][3], A [n][3][3].
 * Backward, from dE/dv or dE/dA: dE/dT (row 0 zero) and dE/da:
 *   vector:  dT_i[1+c][m] = a_i[m] dv_i[c];  da_i[m] = sum_c dv_i[c] T_i[1+c][m]
 *   tensor:  dT_i[1+c][m] = a_i[m] sum_d (dA_i[c][d] + dA_i[d][c]) T_i[1+d][m];
 *            da_i[m] = sum_{c,d} dA_i[c][d] T_i[1+c][m] T_i[1+d][m]
 */
void or_vector_head(const double *T, const double *a, int64_t n, int M, double *v) {
  for (int64_t i = 0; i < n; ++i)
    for (int c = 0; c < 3; ++c) {
      double s = 0.0;
      for (int m = 0; m < M; ++m) s += a[i * M + m] * T[(i * 4 + 1 + c) * M + m];
      v[i * 3 + c] = s;
    }
}

void or_vector_head_grad(const double *T, const double *a, const double *dv, int64_t n, int M, double *dT,
                         double *da) {
  for (int64_t i = 0; i < n; ++i)
    for (int m = 0; m < M; ++m) {
      dT[(i * 4 + 0) * M + m] = 0.0;
      double s = 0.0;
      for (int c = 0; c < 3; ++c) {
        dT[(i * 4 + 1 + c) * M + m] = a[i * M + m] * dv[i * 3 + c];
        s += dv[i * 3 + c] * T[(i * 4 + 1 + c) * M + m];
      }
      da[i * M + m] = s;
    }
}

void or_tensor_head(const double *T, const double *a, int64_t n, int M, double *A) {
  for (int64_t i = 0; i < n; ++i)
    for (int c = 0; c < 3; ++c)
      for (int d = 0; d < 3; ++d) {
        double s = 0.0;
        for (int m = 0; m < M; ++m) s += a[i * M + m] * (T[(i * 4 + 1 + c) * M + m] * T[(i * 4 + 1 + d) * M + m]);
        A[(i * 3 + c) * 3 + d] = s;
      }
}

void or_tensor_head_grad(const double *T, const double *a, const double *dA, int64_t n, int M, double *dT,
                         double *da) {
  for (int64_t i = 0; i < n; ++i)
    for (int m = 0; m < M; ++m) {
      const double *G = dA + i * 9;
      dT[(i * 4 + 0) * M + m] = 0.0;
      double s = 0.0;
      for (int c = 0; c < 3; ++c) {
        double u = 0.0;
        for (int d = 0; d < 3; ++d) {
          const double td = T[(i * 4 + 1 + d) * M + m];
          u += (G[3 * c + d] + G[3 * d + c]) * td;
          s += G[3 * c + d] * T[(i * 4 + 1 + c) * M + m] * td;
        }
        dT[(i * 4 + 1 + c) * M + m] = a[i * M + m] * u;
      }
      da[i * M + m] = s;
    }
}
