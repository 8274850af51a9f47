/*
 * Seed-Q oracle, side-information-free rung schedule (Sec. 3.3 Eq. imp and
 * the floor, Sec. 3.4 hull and Eq. ladder, App. A.5 ties, App. A.7 on
 * encoder/decoder agreement, Alg. 1 allocation steps, Alg. 2 schedule steps).
 * TEST INFRASTRUCTURE ONLY: see seedq_oracle.h.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "seedq_oracle.h"

/* ------------------------- factors of Eq. imp ------------------------- */

static const float *g_sort_key;

static int cmp_index(const void *pa, const void *pb) {
  const int32_t a = *(const int32_t *)pa, b = *(const int32_t *)pb;
  const float va = g_sort_key[a], vb = g_sort_key[b];
  if (va < vb) return -1;
  if (va > vb) return 1;
  return (a > b) - (a < b); /* stable: ties by channel index */
}

int or_factors_init(or_factors *f, int64_t R, int64_t C, const float *a,
                    const float *rho) {
  memset(f, 0, sizeof(*f));
  if (R <= 0 || C <= 0 || (C % 8) != 0) return -1;
  f->R = R;
  f->C = C;
  f->perm = (int32_t *)malloc(sizeof(int32_t) * (size_t)C);
  f->abar = (double *)malloc(sizeof(double) * (size_t)(C / 8));
  f->rho = (double *)malloc(sizeof(double) * (size_t)R);
  if (!f->perm || !f->abar || !f->rho) return -1;

  /* Sec. 3.3: input channels sorted by a before blocking (ascending, stable). */
  for (int64_t c = 0; c < C; ++c) f->perm[c] = (int32_t)c;
  g_sort_key = a;
  qsort(f->perm, (size_t)C, sizeof(int32_t), cmp_index);

  /* Eq. imp: abar_b = (1/B) sum_{j in b} a_j, then unit mean over the tensor. */
  const int64_t nb = C / 8;
  for (int64_t c = 0; c < nb; ++c) {
    double s = 0.0;
    for (int i = 0; i < 8; ++i) s = s + (double)a[f->perm[8 * c + i]];
    f->abar[c] = s / 8.0;
  }
  double sa = 0.0;
  for (int64_t c = 0; c < nb; ++c) sa = sa + f->abar[c];
  const double ma = sa / (double)nb;
  if (!(ma > 0.0)) return -1;
  for (int64_t c = 0; c < nb; ++c) f->abar[c] = f->abar[c] / ma;

  f->rho_uniform = 1;
  if (rho) {
    double sr = 0.0;
    for (int64_t r = 0; r < R; ++r) sr = sr + (double)rho[r];
    const double mr = sr / (double)R;
    if (!(mr > 0.0)) return -1;
    for (int64_t r = 0; r < R; ++r) {
      f->rho[r] = (double)rho[r] / mr;
      if (f->rho[r] != 1.0) f->rho_uniform = 0;
    }
  } else {
    for (int64_t r = 0; r < R; ++r) f->rho[r] = 1.0;
  }
  return 0;
}

void or_factors_free(or_factors *f) {
  free(f->perm);
  free(f->abar);
  free(f->rho);
  memset(f, 0, sizeof(*f));
}

/* Eq. imp times the row factor, then the floor imp <- max(imp, q). */
double or_imp(const or_factors *f, const or_schedule *s, int64_t r, int64_t c) {
  double v = f->abar[c] * f->rho[r];
  if (v < s->q) v = s->q;
  return v;
}

/* Eq. ladder: j(b) = 1 + |{j : lambda/s_j <= imp_b}| (0-based here). */
int or_ladder(const or_schedule *s, double imp) {
  int j = 0;
  for (int i = 0; i < s->J - 1; ++i)
    if (s->theta[i] <= imp) ++j;
  return j;
}

static int is_tied(const or_schedule *s, double imp) {
  return s->j_tie >= 0 && imp == s->theta[s->j_tie];
}

/* Rungs of one row; *remaining is the number of tied blocks still to demote. */
static void rung_row(const or_factors *f, const or_schedule *s, int64_t r,
                     int64_t *remaining, uint8_t *out) {
  const int64_t nb = f->C / 8;
  for (int64_t c = 0; c < nb; ++c) {
    const double imp = or_imp(f, s, r, c);
    int j = or_ladder(s, imp);
    if (is_tied(s, imp) && *remaining > 0) {
      j -= 1;
      *remaining -= 1;
    }
    out[c] = (uint8_t)j;
  }
}

static int64_t tied_in_row(const or_factors *f, const or_schedule *s, int64_t r) {
  int64_t n = 0;
  for (int64_t c = 0; c < f->C / 8; ++c)
    if (is_tied(s, or_imp(f, s, r, c))) ++n;
  return n;
}

int64_t or_tie_remaining(const or_factors *f, const or_schedule *s,
                         int64_t tie_count, int64_t r0) {
  int64_t remaining = tie_count;
  for (int64_t r = 0; r < r0 && remaining > 0; ++r) {
    remaining -= tied_in_row(f, s, r);
    if (remaining < 0) remaining = 0;
  }
  return remaining;
}

void or_rung_rows_cont(const or_factors *f, const or_schedule *s,
                       int64_t *remaining, int64_t r0, int64_t nrows,
                       uint8_t *out) {
  for (int64_t i = 0; i < nrows; ++i)
    rung_row(f, s, r0 + i, remaining, out + i * (f->C / 8));
}

void or_rung_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                  int64_t r0, int64_t nrows, uint8_t *out) {
  int64_t remaining = or_tie_remaining(f, s, tie_count, r0);
  or_rung_rows_cont(f, s, &remaining, r0, nrows, out);
}

int64_t or_tied_blocks(const or_factors *f, const or_schedule *s) {
  int64_t n = 0;
  for (int64_t r = 0; r < f->R; ++r) n += tied_in_row(f, s, r);
  return n;
}

uint64_t or_row_bit_offset(const or_factors *f, const or_schedule *s,
                           int64_t tie_count, int64_t r_end) {
  const int64_t nb = f->C / 8;
  uint8_t *row = (uint8_t *)malloc((size_t)nb);
  int64_t remaining = tie_count;
  uint64_t bits = 0;
  for (int64_t r = 0; r < r_end; ++r) {
    rung_row(f, s, r, &remaining, row);
    for (int64_t c = 0; c < nb; ++c)
      bits += (uint64_t)or_block_bits(s->S[row[c]], s->k[row[c]]);
  }
  free(row);
  return bits;
}

/* ------------------------- hull (Sec. 3.4) ------------------------- */

int or_hull(int n, const int *S, const int *k, const double *e, int *idx) {
  /* Reading R10: keep the lower e among rungs of equal rate. */
  int *cand = (int *)malloc(sizeof(int) * (size_t)n);
  int nc = 0;
  for (int i = 0; i < n; ++i) {
    const int li = or_block_bits(S[i], k[i]);
    int keep = 1;
    for (int j = 0; j < n; ++j) {
      if (j == i || or_block_bits(S[j], k[j]) != li) continue;
      if (e[j] < e[i] || (e[j] == e[i] && j < i)) keep = 0;
    }
    if (keep) cand[nc++] = i;
  }
  /* Sort by rate (insertion sort: a handful of points). */
  for (int a = 1; a < nc; ++a) {
    const int v = cand[a];
    int b = a - 1;
    while (b >= 0 && or_block_bits(S[cand[b]], k[cand[b]]) > or_block_bits(S[v], k[v])) {
      cand[b + 1] = cand[b];
      --b;
    }
    cand[b + 1] = v;
  }
  /* Lower hull by the monotone chain; collinear middle points are dropped. */
  int J = 0;
  for (int a = 0; a < nc; ++a) {
    const int p = cand[a];
    const double px = or_block_bits(S[p], k[p]) / 8.0, py = e[p];
    while (J >= 2) {
      const int o = idx[J - 2], m = idx[J - 1];
      const double ox = or_block_bits(S[o], k[o]) / 8.0, oy = e[o];
      const double mx = or_block_bits(S[m], k[m]) / 8.0, my = e[m];
      const double cross = (mx - ox) * (py - oy) - (my - oy) * (px - ox);
      if (cross <= 0.0) --J;
      else break;
    }
    idx[J++] = p;
  }
  /* A rung past the minimum damage never helps: drop a rising tail. */
  while (J >= 2 && e[idx[J - 1]] >= e[idx[J - 2]]) --J;
  free(cand);
  return J;
}

/* ------------------------- allocator (Alg. 1) ------------------------- */

/* First block c of row r whose floored importance is >= thr (or > thr when
 * strict); imp is non-decreasing in c because abar is (sorted channels). */
static int64_t row_first(const or_factors *f, double q, int64_t r, double thr,
                         int strict) {
  int64_t lo = 0, hi = f->C / 8;
  while (lo < hi) {
    const int64_t mid = lo + (hi - lo) / 2;
    double v = f->abar[mid] * f->rho[r];
    if (v < q) v = q;
    const int pass = strict ? (v > thr) : (v >= thr);
    if (pass) hi = mid;
    else lo = mid + 1;
  }
  return lo;
}

/* Number of blocks of the tensor with raw importance <= v (no floor). */
static uint64_t count_le(const or_factors *f, double v) {
  uint64_t n = 0;
  const int64_t rows = f->rho_uniform ? 1 : f->R;
  for (int64_t r = 0; r < rows; ++r)
    n += (uint64_t)row_first(f, -INFINITY, r, v, 1);
  return f->rho_uniform ? n * (uint64_t)f->R : n;
}

/* Total payload bits of the tensor with thresholds th, tied blocks promoted. */
static uint64_t tensor_bits(const or_factors *f, double q, int J, const int *L,
                            const double *th) {
  const int64_t nb = f->C / 8;
  const int64_t rows = f->rho_uniform ? 1 : f->R;
  uint64_t bits = 0;
  for (int64_t r = 0; r < rows; ++r) {
    uint64_t rb = (uint64_t)L[0] * (uint64_t)nb;
    for (int j = 0; j < J - 1; ++j) {
      const int64_t n_ge = nb - row_first(f, q, r, th[j], 0);
      rb += (uint64_t)(L[j + 1] - L[j]) * (uint64_t)n_ge;
    }
    bits += rb;
  }
  return f->rho_uniform ? bits * (uint64_t)f->R : bits;
}

/* Blocks of the tensor whose floored importance equals v. */
static uint64_t tied_count(const or_factors *f, double q, double v) {
  uint64_t n = 0;
  const int64_t rows = f->rho_uniform ? 1 : f->R;
  for (int64_t r = 0; r < rows; ++r)
    n += (uint64_t)(row_first(f, q, r, v, 1) - row_first(f, q, r, v, 0));
  return f->rho_uniform ? n * (uint64_t)f->R : n;
}

static uint64_t set_bits(int nt, const or_factors *const *f, double q, int J,
                         const int *L, const double *th) {
  uint64_t b = 0;
  for (int t = 0; t < nt; ++t) b += tensor_bits(f[t], q, J, L, th);
  return b;
}

static double from_bits(int64_t p) {
  double d;
  memcpy(&d, &p, sizeof d);
  return d;
}

static int64_t to_bits(double d) {
  int64_t p;
  memcpy(&p, &d, sizeof p);
  return p;
}

static void thresholds(int J, const double *slopes, double lambda, double *th) {
  for (int j = 0; j < J - 1; ++j) th[j] = lambda / slopes[j];
}

int or_allocate(int nt, const or_factors *const *f, int J, const int *S,
                const int *k, const double *slopes, double rbar, double floor_f,
                double *theta, int *j_tie, double *q_out, int64_t *tie_count,
                uint64_t *bits) {
  int L[32];
  double th_lo[32], th_hi[32];
  uint64_t nblocks = 0;
  for (int j = 0; j < J; ++j) L[j] = or_block_bits(S[j], k[j]);
  for (int t = 0; t < nt; ++t) nblocks += (uint64_t)f[t]->R * (uint64_t)(f[t]->C / 8);

  /* Alg. 1: q <- f-quantile of {imp_b}; the m-th smallest value, m = ceil(f N). */
  uint64_t m = (uint64_t)ceil(floor_f * (double)nblocks);
  if (m < 1) m = 1;
  int64_t lo = 0, hi = to_bits(INFINITY);
  while (lo < hi) { /* smallest v (positive doubles order as integers) */
    const int64_t mid = lo + (hi - lo) / 2;
    uint64_t n = 0;
    for (int t = 0; t < nt; ++t) n += count_le(f[t], from_bits(mid));
    if (n >= m) hi = mid;
    else lo = mid + 1;
  }
  const double q = from_bits(lo);
  *q_out = q;

  /* Alg. 1: bisection on lambda for mean payload rate <= rbar. */
  const uint64_t budget = (uint64_t)floor(8.0 * rbar * (double)nblocks);
  thresholds(J, slopes, INFINITY, th_hi);
  if (set_bits(nt, f, q, J, L, th_hi) > budget) return -1; /* infeasible */
  thresholds(J, slopes, 0.0, th_lo);
  if (set_bits(nt, f, q, J, L, th_lo) <= budget) { /* every block on the top rung */
    for (int j = 0; j < J - 1; ++j) theta[j] = th_lo[j];
    *j_tie = -1;
    for (int t = 0; t < nt; ++t) {
      tie_count[t] = 0;
      bits[t] = tensor_bits(f[t], q, J, L, th_lo);
    }
    return 0;
  }
  lo = 0;
  hi = to_bits(INFINITY);
  while (hi - lo > 1) { /* invariant: bits(lo) > budget >= bits(hi) */
    const int64_t mid = lo + (hi - lo) / 2;
    double th[32];
    thresholds(J, slopes, from_bits(mid), th);
    if (set_bits(nt, f, q, J, L, th) > budget) lo = mid;
    else hi = mid;
  }
  thresholds(J, slopes, from_bits(lo), th_lo); /* over budget */
  thresholds(J, slopes, from_bits(hi), th_hi); /* within budget */

  /* The critical tied group: blocks with th_lo[j] <= imp < th_hi[j]. */
  int jt = -1;
  double v = 0.0;
  for (int j = 0; j < J - 1; ++j) {
    double vmin = INFINITY;
    for (int t = 0; t < nt; ++t) {
      const int64_t rows = f[t]->rho_uniform ? 1 : f[t]->R;
      for (int64_t r = 0; r < rows; ++r) {
        const int64_t c = row_first(f[t], q, r, th_lo[j], 0);
        if (c < f[t]->C / 8) {
          double x = f[t]->abar[c] * f[t]->rho[r];
          if (x < q) x = q;
          if (x < vmin) vmin = x;
        }
      }
    }
    if (vmin < th_hi[j]) {
      if (jt >= 0) return -2; /* two groups straddle at once: not expected */
      jt = j;
      v = vmin;
    }
  }
  if (jt < 0) return -3;
  for (int j = 0; j < J - 1; ++j) theta[j] = th_hi[j];
  theta[jt] = v;
  const uint64_t b_hi = set_bits(nt, f, q, J, L, theta);
  const uint64_t step = (uint64_t)(L[jt + 1] - L[jt]);
  const uint64_t excess = b_hi > budget ? b_hi - budget : 0;
  uint64_t T = (excess + step - 1) / step;
  /* App. A.5: demote members of the group in block order until the budget is
   * met exactly (tensor order, then row-major order within a tensor). */
  for (int t = 0; t < nt; ++t) {
    const uint64_t tied = T ? tied_count(f[t], q, v) : 0;
    const uint64_t d = T < tied ? T : tied;
    tie_count[t] = (int64_t)d;
    T -= d;
    bits[t] = tensor_bits(f[t], q, J, L, theta) - d * step;
  }
  if (T != 0) return -4;
  *j_tie = jt;
  return 0;
}
