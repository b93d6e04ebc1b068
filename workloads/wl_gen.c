/*
 * Seeded synthetic inputs for the DP Compress tabulate-fusion path.
 *
 * This file only MAKES INPUTS: random numbers, geometries (random neighbour
 * shells, jittered fcc lattices, rigid water), neighbour lists sorted by
 * neighbour type and then by distance with per-type caps sel_alpha, and the
 * rows of the environment matrix built from them (paper, Sec. II, the
 * weighting function s(r) and the 4-vector rows of R~).  It holds none of the
 * method's arithmetic: no embedding net, no table, no interval search, no
 * fused contraction.  Both the CUDA path and the oracle consume its output.
 *
 * Determinism: every random number comes from splitmix64 (Steele, Lea and
 * Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014), and
 * the only transcendental functions used (log for the polar normal method,
 * cos for the cosine switch) are computed here from their series so that the
 * x86-64 and aarch64 builds produce the same bits.  Build with
 * -ffp-contract=off.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ RNG */

static uint64_t sm64_next(uint64_t *state) {
  uint64_t z = (*state += 0x9E3779B97F4A7C15ULL);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* uniform on [0, 1) with 53 random bits */
static double u01(uint64_t *st) { return (double)(sm64_next(st) >> 11) * 0x1.0p-53; }

/* natural log from frexp + the atanh series; x > 0 */
static double det_log(double x) {
  int e;
  double m = frexp(x, &e); /* x = m * 2^e, m in [0.5, 1) */
  if (m < 0.70710678118654752440) {
    m *= 2.0;
    e -= 1;
  }
  double z = (m - 1.0) / (m + 1.0), z2 = z * z, term = z, sum = 0.0;
  for (int k = 1; k <= 45; k += 2) {
    sum += term / (double)k;
    term *= z2;
  }
  return 2.0 * sum + (double)e * 0.69314718055994530942;
}

/* sin on [-pi/2, pi/2] from its Taylor series */
static double det_sin_reduced(double y) {
  double y2 = y * y, term = y, sum = 0.0;
  for (int k = 1; k <= 31; k += 2) {
    sum += term;
    term *= -y2 / ((double)(k + 1) * (double)(k + 2));
  }
  return sum;
}

static const double WL_PI = 3.14159265358979323846;

/* cos on [0, pi]: cos(x) = -sin(x - pi/2) */
static double det_cos_0pi(double x) { return -det_sin_reduced(x - 0.5 * WL_PI); }

typedef struct {
  uint64_t st;
  int has_spare;
  double spare;
} nrng_t;

/* standard normal by Marsaglia's polar method */
static double nrm(nrng_t *g) {
  if (g->has_spare) {
    g->has_spare = 0;
    return g->spare;
  }
  double u, v, q;
  do {
    u = 2.0 * u01(&g->st) - 1.0;
    v = 2.0 * u01(&g->st) - 1.0;
    q = u * u + v * v;
  } while (q >= 1.0 || q == 0.0);
  double f = sqrt(-2.0 * det_log(q) / q);
  g->spare = v * f;
  g->has_spare = 1;
  return u * f;
}

static void nrng_init(nrng_t *g, uint64_t seed) {
  g->st = seed * 0x2545F4914F6CDD1DULL + 0x1234567ULL;
  g->has_spare = 0;
  g->spare = 0.0;
  (void)sm64_next(&g->st);
}

/* uniform direction on the unit sphere: a normalised 3-d normal vector */
static void rand_dir(nrng_t *g, double d[3]) {
  double n2;
  do {
    d[0] = nrm(g);
    d[1] = nrm(g);
    d[2] = nrm(g);
    n2 = d[0] * d[0] + d[1] * d[1] + d[2] * d[2];
  } while (n2 < 1e-12);
  double inv = 1.0 / sqrt(n2);
  d[0] *= inv;
  d[1] *= inv;
  d[2] *= inv;
}

/* ------------------------------------------------------------ exported */

void wl_normal(uint64_t seed, int64_t n, double mean, double std, double *out) {
  nrng_t g;
  nrng_init(&g, seed);
  for (int64_t k = 0; k < n; ++k) out[k] = mean + std * nrm(&g);
}

void wl_uniform(uint64_t seed, int64_t n, double lo, double hi, double *out) {
  uint64_t st = seed * 0x9E3779B97F4A7C15ULL + 77ULL;
  (void)sm64_next(&st);
  for (int64_t k = 0; k < n; ++k) out[k] = lo + (hi - lo) * u01(&st);
}

/* Test hook: expose the deterministic log / cos so tests can check them. */
double wl_det_log(double x) { return det_log(x); }
double wl_det_cos(double x) { return det_cos_0pi(x); }

/*
 * Weighting function s(r).  kind 0: cosine switch used by the workloads,
 *   s = 1/r                                   r < rcs
 *   s = (1/r) (0.5 cos(pi (r-rcs)/(rc-rcs)) + 0.5)   rcs <= r < rc
 *   s = 0                                     r >= rc
 * kind 1: the paper's quintic switch (Sec. II, the weighting-function
 * equation), u^3 (-6u^2 + 15u - 10) + 1 in place of the cosine.
 */
double wl_switch(double r, double rcs, double rc, int kind) {
  if (r < rcs) return 1.0 / r;
  if (r >= rc) return 0.0;
  double u = (r - rcs) / (rc - rcs);
  double w;
  if (kind == 1)
    w = u * u * u * (-6.0 * u * u + 15.0 * u - 10.0) + 1.0;
  else
    w = 0.5 * det_cos_0pi(WL_PI * u) + 0.5;
  return w / r;
}

/*
 * Random neighbour shells (the "tiny" workload): every atom gets nreal
 * neighbours at r ~ U[rmin, rmax), uniform directions, sorted by r; rows
 * nreal..sel-1 are zero padding.  One neighbour type.
 */
int wl_random_shell(uint64_t seed, int nloc, int nreal, int sel, double rmin, double rmax, double rcs,
                    double rc, int kind, double *s, double *Rt, int32_t *nvalid) {
  if (nloc < 0 || nreal < 0 || nreal > sel) return -1;
  nrng_t g;
  nrng_init(&g, seed);
  double *r = (double *)malloc(sizeof(double) * (nreal > 0 ? nreal : 1));
  double *dir = (double *)malloc(sizeof(double) * 3 * (nreal > 0 ? nreal : 1));
  if (!r || !dir) {
    free(r);
    free(dir);
    return -2;
  }
  for (int i = 0; i < nloc; ++i) {
    for (int j = 0; j < nreal; ++j) {
      r[j] = rmin + (rmax - rmin) * u01(&g.st);
      rand_dir(&g, dir + 3 * j);
    }
    /* insertion sort by distance (stable) */
    for (int a = 1; a < nreal; ++a) {
      double rv = r[a], d0 = dir[3 * a], d1 = dir[3 * a + 1], d2 = dir[3 * a + 2];
      int b = a - 1;
      while (b >= 0 && r[b] > rv) {
        r[b + 1] = r[b];
        dir[3 * (b + 1)] = dir[3 * b];
        dir[3 * (b + 1) + 1] = dir[3 * b + 1];
        dir[3 * (b + 1) + 2] = dir[3 * b + 2];
        --b;
      }
      r[b + 1] = rv;
      dir[3 * (b + 1)] = d0;
      dir[3 * (b + 1) + 1] = d1;
      dir[3 * (b + 1) + 2] = d2;
    }
    for (int j = 0; j < sel; ++j) {
      int64_t row = (int64_t)i * sel + j;
      if (j < nreal) {
        double sv = wl_switch(r[j], rcs, rc, kind);
        s[row] = sv;
        Rt[4 * row + 0] = sv;
        Rt[4 * row + 1] = sv * dir[3 * j + 0];
        Rt[4 * row + 2] = sv * dir[3 * j + 1];
        Rt[4 * row + 3] = sv * dir[3 * j + 2];
      } else {
        s[row] = 0.0;
        Rt[4 * row + 0] = Rt[4 * row + 1] = Rt[4 * row + 2] = Rt[4 * row + 3] = 0.0;
      }
    }
    nvalid[i] = nreal;
  }
  free(r);
  free(dir);
  return 0;
}

/* wrap x into [0, L) */
static double wrap(double x, double L) {
  double y = fmod(x, L);
  if (y < 0.0) y += L;
  if (y >= L) y -= L;
  return y;
}

/* jittered fcc lattice of nx*ny*nz cubic cells (4 atoms each), periodic box */
int wl_fcc(uint64_t seed, int nx, int ny, int nz, double a, double jitter, double *pos, double box[3]) {
  static const double basis[4][3] = {{0, 0, 0}, {0.5, 0.5, 0}, {0.5, 0, 0.5}, {0, 0.5, 0.5}};
  nrng_t g;
  nrng_init(&g, seed);
  box[0] = nx * a;
  box[1] = ny * a;
  box[2] = nz * a;
  int64_t k = 0;
  for (int ix = 0; ix < nx; ++ix)
    for (int iy = 0; iy < ny; ++iy)
      for (int iz = 0; iz < nz; ++iz)
        for (int b = 0; b < 4; ++b) {
          double p0 = (ix + basis[b][0]) * a + jitter * nrm(&g);
          double p1 = (iy + basis[b][1]) * a + jitter * nrm(&g);
          double p2 = (iz + basis[b][2]) * a + jitter * nrm(&g);
          pos[3 * k + 0] = wrap(p0, box[0]);
          pos[3 * k + 1] = wrap(p1, box[1]);
          pos[3 * k + 2] = wrap(p2, box[2]);
          ++k;
        }
  return 0;
}

/* species by independent draws: type t with probability frac[t] */
void wl_species(uint64_t seed, int64_t n, int ntypes, const double *frac, int32_t *types) {
  uint64_t st = seed * 0xD1342543DE82EF95ULL + 99ULL;
  (void)sm64_next(&st);
  for (int64_t k = 0; k < n; ++k) {
    double u = u01(&st), acc = 0.0;
    int t = ntypes - 1;
    for (int q = 0; q < ntypes; ++q) {
      acc += frac[q];
      if (u < acc) {
        t = q;
        break;
      }
    }
    types[k] = t;
  }
}

/*
 * Rigid water: nmol oxygens placed uniformly in a periodic cube of side L by
 * random sequential addition, rejecting any O closer than r_oo_min to an
 * existing O; each O gets two H at r_oh with H-O-H angle theta_deg in a
 * random orientation.  extra_o further oxygens (no H) are added the same
 * way.  Output order: all O (type 0), then all H (type 1).
 * Returns the number of attempts, or a negative error.
 */
int64_t wl_water(uint64_t seed, int nmol, int extra_o, double L, double r_oo_min, double r_oh,
                 double theta_deg, double *pos, int32_t *types) {
  int no = nmol + extra_o;
  int nc = (int)floor(L / r_oo_min);
  if (nc < 1) nc = 1;
  double cs = L / nc;
  const int CAP = 24;
  int64_t ncell = (int64_t)nc * nc * nc;
  int32_t *cnt = (int32_t *)calloc((size_t)ncell, sizeof(int32_t));
  int32_t *lst = (int32_t *)malloc(sizeof(int32_t) * (size_t)ncell * CAP);
  if (!cnt || !lst) {
    free(cnt);
    free(lst);
    return -2;
  }
  nrng_t g;
  nrng_init(&g, seed);
  double rmin2 = r_oo_min * r_oo_min;
  int64_t attempts = 0;
  for (int k = 0; k < no; ++k) {
    for (;;) {
      if (++attempts > (int64_t)no * 2000) {
        free(cnt);
        free(lst);
        return -3;
      }
      double p[3] = {L * u01(&g.st), L * u01(&g.st), L * u01(&g.st)};
      int c[3];
      for (int d = 0; d < 3; ++d) {
        c[d] = (int)(p[d] / cs);
        if (c[d] >= nc) c[d] = nc - 1;
      }
      int ok = 1;
      for (int dx = -1; dx <= 1 && ok; ++dx)
        for (int dy = -1; dy <= 1 && ok; ++dy)
          for (int dz = -1; dz <= 1 && ok; ++dz) {
            int cx = ((c[0] + dx) % nc + nc) % nc, cy = ((c[1] + dy) % nc + nc) % nc,
                cz = ((c[2] + dz) % nc + nc) % nc;
            int64_t ci = ((int64_t)cx * nc + cy) * nc + cz;
            for (int q = 0; q < cnt[ci]; ++q) {
              int o = lst[ci * CAP + q];
              double r2 = 0.0;
              for (int d = 0; d < 3; ++d) {
                double dd = pos[3 * o + d] - p[d];
                dd -= L * nearbyint(dd / L);
                r2 += dd * dd;
              }
              if (r2 < rmin2) {
                ok = 0;
                break;
              }
            }
          }
      if (!ok) continue;
      int64_t ci = ((int64_t)c[0] * nc + c[1]) * nc + c[2];
      if (cnt[ci] >= CAP) continue;
      lst[ci * CAP + cnt[ci]++] = k;
      pos[3 * k + 0] = p[0];
      pos[3 * k + 1] = p[1];
      pos[3 * k + 2] = p[2];
      types[k] = 0;
      break;
    }
  }
  free(cnt);
  free(lst);
  /* hydrogens */
  double half = 0.5 * theta_deg * WL_PI / 180.0;
  double ch = det_cos_0pi(half), sh = det_cos_0pi(0.5 * WL_PI - half);
  for (int k = 0; k < nmol; ++k) {
    double u1[3], v[3], u2[3];
    rand_dir(&g, u1);
    double n2;
    do {
      rand_dir(&g, v);
      double dot = v[0] * u1[0] + v[1] * u1[1] + v[2] * u1[2];
      for (int d = 0; d < 3; ++d) u2[d] = v[d] - dot * u1[d];
      n2 = u2[0] * u2[0] + u2[1] * u2[1] + u2[2] * u2[2];
    } while (n2 < 1e-6);
    double inv = 1.0 / sqrt(n2);
    for (int d = 0; d < 3; ++d) u2[d] *= inv;
    for (int h = 0; h < 2; ++h) {
      int64_t idx = no + 2 * (int64_t)k + h;
      double sgn = h == 0 ? 1.0 : -1.0;
      for (int d = 0; d < 3; ++d) pos[3 * idx + d] = wrap(pos[3 * k + d] + r_oh * (ch * u1[d] + sgn * sh * u2[d]), L);
      types[idx] = 1;
    }
  }
  return attempts;
}

/* ------------------------------------------------------- neighbour list */

typedef struct {
  double r, d[3];
  int32_t j, t;
  int8_t sh[3];
} cand_t;

static int cand_cmp(const void *pa, const void *pb) {
  const cand_t *a = (const cand_t *)pa, *b = (const cand_t *)pb;
  if (a->t != b->t) return a->t < b->t ? -1 : 1;
  if (a->r != b->r) return a->r < b->r ? -1 : 1;
  return a->j < b->j ? -1 : (a->j > b->j ? 1 : 0);
}

/*
 * Environment-matrix rows for every atom (paper, Sec. II): neighbours within
 * rc under the minimum-image convention, grouped by neighbour type, sorted
 * by distance inside each group, capped at sel[t] (the nearest are kept),
 * zero rows after the last real neighbour of each group.  Row of neighbour
 * j: s = s(r_ij), R~ = (s, s x/r, s y/r, s z/r) with (x, y, z) = r_j - r_i.
 * Optional normalisation (paper, Sec. II): when norm != NULL the rows become
 * ((s - norm[0]) / norm[1], s x/r / norm[2], ...), with norm = {mean_s,
 * std_s, std_all}, and the s column gets the same map.  Padding rows stay 0.
 *
 * stats (int64[4]): total real neighbours before the cap, rows dropped by
 * the cap, maximum per-atom real count, rows kept.
 * srange (double[2]): min and max of s over kept rows.
 * nlist (int32 [natoms][nnei], optional): the neighbour index of each row,
 * -1 on padding rows; shift (int8 [natoms][nnei][3], optional): the periodic
 * image of that neighbour, r_j + shift * box being the position the row uses.
 */
int wl_envmat(int64_t natoms, const double *pos, const int32_t *types, const double box[3], int ntypes,
              const int32_t *sel, double rcs, double rc, int kind, const double *norm, double *s, double *Rt,
              int32_t *nvalid, int64_t *stats, double *srange, int nthreads, int32_t *nlist, int8_t *shift) {
  if (ntypes < 1 || ntypes > 64) return -1;
  for (int d = 0; d < 3; ++d)
    if (box[d] < 2.0 * rc) return -4; /* minimum image needs L >= 2 rc */
  int nnei = 0;
  int off[65];
  for (int t = 0; t < ntypes; ++t) {
    off[t] = nnei;
    nnei += sel[t];
  }
  int nc[3];
  double cs[3];
  for (int d = 0; d < 3; ++d) {
    nc[d] = (int)floor(box[d] / rc);
    if (nc[d] < 1) nc[d] = 1;
    cs[d] = box[d] / nc[d];
  }
  int64_t ncell = (int64_t)nc[0] * nc[1] * nc[2];
  int32_t *head = (int32_t *)malloc(sizeof(int32_t) * (size_t)ncell);
  int32_t *next = (int32_t *)malloc(sizeof(int32_t) * (size_t)(natoms > 0 ? natoms : 1));
  int32_t *cell_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)(natoms > 0 ? natoms : 1));
  if (!head || !next || !cell_of) {
    free(head);
    free(next);
    free(cell_of);
    return -2;
  }
  for (int64_t c = 0; c < ncell; ++c) head[c] = -1;
  int32_t maxocc = 0;
  int32_t *occ = (int32_t *)calloc((size_t)ncell, sizeof(int32_t));
  for (int64_t a = natoms - 1; a >= 0; --a) {
    int c[3];
    for (int d = 0; d < 3; ++d) {
      c[d] = (int)(pos[3 * a + d] / cs[d]);
      if (c[d] >= nc[d]) c[d] = nc[d] - 1;
      if (c[d] < 0) c[d] = 0;
    }
    int64_t ci = ((int64_t)c[0] * nc[1] + c[1]) * nc[2] + c[2];
    cell_of[a] = (int32_t)ci;
    next[a] = head[ci];
    head[ci] = (int32_t)a;
    if (++occ[ci] > maxocc) maxocc = occ[ci];
  }
  free(occ);
  /* unique neighbour-cell offsets per dimension (handles nc < 3) */
  int offs[3][3], noff[3];
  for (int d = 0; d < 3; ++d) {
    noff[d] = 0;
    for (int k = -1; k <= 1; ++k) {
      int v = ((k % nc[d]) + nc[d]) % nc[d];
      int dup = 0;
      for (int q = 0; q < noff[d]; ++q)
        if (((offs[d][q] % nc[d]) + nc[d]) % nc[d] == v) dup = 1;
      if (!dup) offs[d][noff[d]++] = k;
    }
  }
  int64_t capacity = (int64_t)maxocc * 27 + 1;
  int64_t tot_real = 0, tot_drop = 0, max_real = 0, tot_kept = 0;
  double smin = INFINITY, smax = -INFINITY;
  int err = 0;
#ifdef _OPENMP
  if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel num_threads(nthreads) reduction(+ : tot_real, tot_drop, tot_kept) reduction(max : max_real) \
    reduction(min : smin) reduction(max : smax)
#endif
  {
    cand_t *cand = (cand_t *)malloc(sizeof(cand_t) * (size_t)capacity);
    if (!cand) err = 1;
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 256)
#endif
    for (int64_t i = 0; i < natoms; ++i) {
      if (!cand) continue;
      int64_t ci = cell_of[i];
      int c0 = (int)(ci / ((int64_t)nc[1] * nc[2])), c1 = (int)((ci / nc[2]) % nc[1]), c2 = (int)(ci % nc[2]);
      int64_t nca = 0;
      for (int a = 0; a < noff[0]; ++a)
        for (int b = 0; b < noff[1]; ++b)
          for (int e = 0; e < noff[2]; ++e) {
            int x = ((c0 + offs[0][a]) % nc[0] + nc[0]) % nc[0];
            int y = ((c1 + offs[1][b]) % nc[1] + nc[1]) % nc[1];
            int z = ((c2 + offs[2][e]) % nc[2] + nc[2]) % nc[2];
            int64_t cj = ((int64_t)x * nc[1] + y) * nc[2] + z;
            for (int32_t j = head[cj]; j >= 0; j = next[j]) {
              if (j == i) continue;
              double dv[3], r2 = 0.0;
              int8_t sh[3];
              for (int d = 0; d < 3; ++d) {
                double dd = pos[3 * j + d] - pos[3 * i + d];
                const double k = nearbyint(dd / box[d]);
                dd -= box[d] * k;
                sh[d] = (int8_t)(-k);
                dv[d] = dd;
                r2 += dd * dd;
              }
              if (r2 >= rc * rc) continue;
              cand_t cd;
              cd.sh[0] = sh[0];
              cd.sh[1] = sh[1];
              cd.sh[2] = sh[2];
              cd.r = sqrt(r2);
              cd.d[0] = dv[0];
              cd.d[1] = dv[1];
              cd.d[2] = dv[2];
              cd.j = j;
              cd.t = types[j];
              cand[nca++] = cd;
            }
          }
      qsort(cand, (size_t)nca, sizeof(cand_t), cand_cmp);
      tot_real += nca;
      if (nca > max_real) max_real = nca;
      int64_t k = 0;
      for (int t = 0; t < ntypes; ++t) {
        int kept = 0;
        for (; k < nca && cand[k].t == t; ++k) {
          if (kept >= sel[t]) {
            ++tot_drop;
            continue;
          }
          int64_t row = i * nnei + off[t] + kept;
          double r = cand[k].r;
          double sv = wl_switch(r, rcs, rc, kind);
          double sh = sv, sx = sv * cand[k].d[0] / r, sy = sv * cand[k].d[1] / r, sz = sv * cand[k].d[2] / r;
          if (norm) {
            sh = (sv - norm[0]) / norm[1];
            sx /= norm[2];
            sy /= norm[2];
            sz /= norm[2];
          }
          s[row] = sh;
          Rt[4 * row + 0] = sh;
          Rt[4 * row + 1] = sx;
          Rt[4 * row + 2] = sy;
          Rt[4 * row + 3] = sz;
          if (nlist) nlist[row] = cand[k].j;
          if (shift) {
            shift[3 * row + 0] = cand[k].sh[0];
            shift[3 * row + 1] = cand[k].sh[1];
            shift[3 * row + 2] = cand[k].sh[2];
          }
          if (sh < smin) smin = sh;
          if (sh > smax) smax = sh;
          ++kept;
        }
        for (int q = kept; q < sel[t]; ++q) {
          int64_t row = i * nnei + off[t] + q;
          s[row] = 0.0;
          Rt[4 * row + 0] = Rt[4 * row + 1] = Rt[4 * row + 2] = Rt[4 * row + 3] = 0.0;
          if (nlist) nlist[row] = -1;
          if (shift) shift[3 * row + 0] = shift[3 * row + 1] = shift[3 * row + 2] = 0;
        }
        nvalid[i * ntypes + t] = kept;
        tot_kept += kept;
      }
    }
    free(cand);
  }
  free(head);
  free(next);
  free(cell_of);
  if (err) return -2;
  stats[0] = tot_real;
  stats[1] = tot_drop;
  stats[2] = max_real;
  stats[3] = tot_kept;
  srange[0] = smin;
  srange[1] = smax;
  return 0;
}
