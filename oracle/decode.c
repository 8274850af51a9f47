/*
 * Seed-Q oracle, decoder (Alg. 2), fp64 matrix-vector product, synthetic
 * payload packer.  TEST INFRASTRUCTURE ONLY: see seedq_oracle.h.
 */
#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

#include "seedq_oracle.h"

/* IEEE binary16 bit pattern to float, written out from the format definition. */
static float half_to_float(uint16_t h) {
  const int sign = (h >> 15) & 1;
  const int expo = (h >> 10) & 31;
  const int mant = h & 1023;
  double v;
  if (expo == 0) v = ldexp((double)mant, -24);               /* subnormal */
  else if (expo == 31) v = mant ? NAN : INFINITY;
  else v = ldexp(1.0 + (double)mant / 1024.0, expo - 15);
  return (float)(sign ? -v : v);
}

/* bfloat16 is the top half of a binary32 pattern. */
static double bf16_to_double(uint16_t b) {
  const uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static int sign_extend4(uint64_t v) { return (int)(v & 15u) - ((v & 8u) ? 16 : 0); }

int or_decode_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                   const uint8_t *stream, uint64_t stream_bits,
                   const uint32_t *taps, int n_out, const int32_t *outlier_cols,
                   const uint16_t *outlier_vals, int64_t r0, int64_t nrows,
                   float *W) {
  const int64_t C = f->C, nb = C / 8;
  uint8_t *rungs = (uint8_t *)malloc((size_t)nb);
  uint64_t pos = or_row_bit_offset(f, s, tie_count, r0);
  int64_t remaining = or_tie_remaining(f, s, tie_count, r0);
  int rc = 0;
  for (int64_t i = 0; i < nrows && rc == 0; ++i) {
    const int64_t r = r0 + i;
    or_rung_rows_cont(f, s, &remaining, r, 1, rungs);
    float *row = W + i * C;
    for (int64_t c = 0; c < nb; ++c) {
      const int S = s->S[rungs[c]], k = s->k[rungs[c]];
      const int L = or_block_bits(S, k);
      if (pos + (uint64_t)L > stream_bits) { rc = -1; break; }
      /* Read l(g_b) bits: seed, shared exponent, k mantissas (reading R4). */
      const uint32_t seed = (uint32_t)or_read_bits(stream, pos, S);
      const int E = sign_extend4(or_read_bits(stream, pos + (uint64_t)S, 4));
      int t[6];
      for (int j = 0; j < k; ++j)
        t[j] = sign_extend4(or_read_bits(stream, pos + (uint64_t)(S + 4 + 4 * j), 4));
      pos += (uint64_t)L;
      float w[8];
      or_reconstruct_block(S, k, taps[S], seed, E, t, w);
      /* Inverse column permutation: block c holds channels perm[8c..8c+7]. */
      for (int q = 0; q < 8; ++q) row[f->perm[8 * c + q]] = w[q];
    }
    /* Outlier columns overwrite the codec's reconstruction. */
    for (int o = 0; o < n_out; ++o)
      row[outlier_cols[o]] = half_to_float(outlier_vals[r * n_out + o]);
  }
  free(rungs);
  return rc;
}

void or_gemv_f64(int64_t nrows, int64_t C, const float *W, int nb,
                 const uint16_t *x_bf16, double *y) {
  for (int b = 0; b < nb; ++b)
    for (int64_t r = 0; r < nrows; ++r) {
      double acc = 0.0;
      for (int64_t c = 0; c < C; ++c)
        acc = acc + (double)W[r * C + c] * bf16_to_double(x_bf16[b * C + c]);
      y[b * nrows + r] = acc;
    }
}

/* ---------------- threaded baseline timing ---------------- */

typedef struct {
  const or_factors *f;
  const or_schedule *s;
  const uint8_t *stream;
  const uint32_t *taps;
  const uint8_t *rungs;   /* R x nb */
  const uint64_t *offs;   /* R + 1 */
  const uint16_t *x;
  double *y;
  int nb;
  int64_t r0, r1;
} job_t;

static void *job_run(void *arg) {
  job_t *jb = (job_t *)arg;
  const int64_t C = jb->f->C, nblk = C / 8;
  float *row = (float *)malloc(sizeof(float) * (size_t)C);
  for (int64_t r = jb->r0; r < jb->r1; ++r) {
    uint64_t pos = jb->offs[r];
    for (int64_t c = 0; c < nblk; ++c) {
      const int g = jb->rungs[r * nblk + c];
      const int S = jb->s->S[g], k = jb->s->k[g];
      const uint32_t seed = (uint32_t)or_read_bits(jb->stream, pos, S);
      const int E = sign_extend4(or_read_bits(jb->stream, pos + (uint64_t)S, 4));
      int t[6];
      for (int j = 0; j < k; ++j)
        t[j] = sign_extend4(or_read_bits(jb->stream, pos + (uint64_t)(S + 4 + 4 * j), 4));
      pos += (uint64_t)or_block_bits(S, k);
      float w[8];
      or_reconstruct_block(S, k, jb->taps[S], seed, E, t, w);
      for (int q = 0; q < 8; ++q) row[jb->f->perm[8 * c + q]] = w[q];
    }
    for (int b = 0; b < jb->nb; ++b) {
      double acc = 0.0;
      for (int64_t c = 0; c < C; ++c)
        acc = acc + (double)row[c] * bf16_to_double(jb->x[b * C + c]);
      jb->y[b * jb->f->R + r] = acc;
    }
  }
  free(row);
  return NULL;
}

int or_decode_gemv_threads(const or_factors *f, const or_schedule *s,
                           int64_t tie_count, const uint8_t *stream,
                           uint64_t stream_bits, const uint32_t *taps, int nb,
                           const uint16_t *x_bf16, int64_t r0, int64_t nrows,
                           double *y, int nthreads) {
  const int64_t R = r0 + nrows, nblk = f->C / 8;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  uint8_t *rungs = (uint8_t *)malloc((size_t)(R * nblk));
  uint64_t *offs = (uint64_t *)malloc(sizeof(uint64_t) * (size_t)(R + 1));
  or_rung_rows(f, s, tie_count, 0, R, rungs);
  offs[0] = 0;
  for (int64_t r = 0; r < R; ++r) {
    uint64_t b = 0;
    for (int64_t c = 0; c < nblk; ++c) {
      const int g = rungs[r * nblk + c];
      b += (uint64_t)or_block_bits(s->S[g], s->k[g]);
    }
    offs[r + 1] = offs[r] + b;
  }
  if (offs[R] > stream_bits) { free(rungs); free(offs); return -1; }
  pthread_t th[256];
  job_t jobs[256];
  for (int i = 0; i < nthreads; ++i) {
    jobs[i] = (job_t){f, s, stream, taps, rungs, offs, x_bf16, y, nb,
                      r0 + nrows * i / nthreads, r0 + nrows * (i + 1) / nthreads};
    pthread_create(&th[i], NULL, job_run, &jobs[i]);
  }
  for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
  free(rungs);
  free(offs);
  return nthreads;
}

/* ---------------- synthetic stream packer ---------------- */

uint64_t or_synth_pack(const or_factors *f, const or_schedule *s,
                       int64_t tie_count, uint64_t key, uint8_t *stream) {
  const int64_t nb = f->C / 8;
  uint8_t *rungs = (uint8_t *)malloc((size_t)nb);
  int64_t remaining = tie_count;
  uint64_t pos = 0;
  for (int64_t r = 0; r < f->R; ++r) {
    or_rung_rows_cont(f, s, &remaining, r, 1, rungs);
    for (int64_t c = 0; c < nb; ++c) {
      const int S = s->S[rungs[c]], k = s->k[rungs[c]];
      uint32_t seed;
      int E, t[6];
      or_synth_fields(key, (uint64_t)(r * nb + c), S, k, &seed, &E, t);
      or_write_bits(stream, pos, S, seed);
      or_write_bits(stream, pos + (uint64_t)S, 4, (uint64_t)(E & 15));
      for (int j = 0; j < k; ++j)
        or_write_bits(stream, pos + (uint64_t)(S + 4 + 4 * j), 4, (uint64_t)(t[j] & 15));
      pos += (uint64_t)or_block_bits(S, k);
    }
  }
  free(rungs);
  return pos;
}

/* Rows [r0, r0+nrows) of a synthetic tensor computed straight from its block
 * fields (no stream): the same values or_decode_rows gives on the stream that
 * or_synth_pack writes.  Used for sampled rows of tensors too large to pack
 * on the host. */
void or_synth_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                   uint64_t key, const uint32_t *taps, int n_out,
                   const int32_t *outlier_cols, const uint16_t *outlier_vals,
                   int64_t r0, int64_t nrows, float *W) {
  const int64_t C = f->C, nb = C / 8;
  uint8_t *rungs = (uint8_t *)malloc((size_t)nb);
  int64_t remaining = or_tie_remaining(f, s, tie_count, r0);
  for (int64_t i = 0; i < nrows; ++i) {
    const int64_t r = r0 + i;
    or_rung_rows_cont(f, s, &remaining, r, 1, rungs);
    float *row = W + i * C;
    for (int64_t c = 0; c < nb; ++c) {
      const int S = s->S[rungs[c]], k = s->k[rungs[c]];
      uint32_t seed;
      int E, t[6];
      or_synth_fields(key, (uint64_t)(r * nb + c), S, k, &seed, &E, t);
      float w[8];
      or_reconstruct_block(S, k, taps[S], seed, E, t, w);
      for (int q = 0; q < 8; ++q) row[f->perm[8 * c + q]] = w[q];
    }
    for (int o = 0; o < n_out; ++o)
      row[outlier_cols[o]] = half_to_float(outlier_vals[r * n_out + o]);
  }
  free(rungs);
}

/* ---------------- threaded fp64 product straight from synthetic fields ---------------- */

typedef struct {
  const or_factors *f;
  const or_schedule *s;
  int64_t tie_count;
  uint64_t key;
  const uint32_t *taps;
  const uint16_t *x;
  double *y, *yabs;
  int nb;
  int64_t r0, r1;
} sjob_t;

static void *sjob_run(void *arg) {
  sjob_t *jb = (sjob_t *)arg;
  const int64_t C = jb->f->C;
  float *row = (float *)malloc(sizeof(float) * (size_t)C);
  for (int64_t r = jb->r0; r < jb->r1; ++r) {
    or_synth_rows(jb->f, jb->s, jb->tie_count, jb->key, jb->taps, 0, NULL, NULL, r, 1, row);
    for (int b = 0; b < jb->nb; ++b) {
      double acc = 0.0, aab = 0.0;
      for (int64_t c = 0; c < C; ++c) {
        const double xv = bf16_to_double(jb->x[b * C + c]);
        acc = acc + (double)row[c] * xv;
        aab = aab + fabs((double)row[c]) * fabs(xv);
      }
      jb->y[b * jb->f->R + r] = acc;
      if (jb->yabs) jb->yabs[b * jb->f->R + r] = aab;
    }
  }
  free(row);
  return NULL;
}

int or_synth_gemv_threads(const or_factors *f, const or_schedule *s, int64_t tie_count,
                          uint64_t key, const uint32_t *taps, int nb,
                          const uint16_t *x_bf16, int64_t r0, int64_t nrows, double *y,
                          double *yabs, int nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  sjob_t jobs[256];
  for (int i = 0; i < nthreads; ++i) {
    jobs[i] = (sjob_t){f, s, tie_count, key, taps, x_bf16, y, yabs, nb,
                       r0 + nrows * i / nthreads, r0 + nrows * (i + 1) / nthreads};
    pthread_create(&th[i], NULL, sjob_run, &jobs[i]);
  }
  for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
  return nthreads;
}

/* Pack rows [r0, r0+nrows) of the synthetic stream into out starting at bit 0
 * (zeroed by the caller).  Returns the number of bits written. */
uint64_t or_synth_pack_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                            uint64_t key, int64_t r0, int64_t nrows, uint8_t *out) {
  const int64_t nb = f->C / 8;
  uint8_t *rungs = (uint8_t *)malloc((size_t)nb);
  int64_t remaining = or_tie_remaining(f, s, tie_count, r0);
  uint64_t pos = 0;
  for (int64_t r = r0; r < r0 + nrows; ++r) {
    or_rung_rows_cont(f, s, &remaining, r, 1, rungs);
    for (int64_t c = 0; c < nb; ++c) {
      const int S = s->S[rungs[c]], k = s->k[rungs[c]];
      uint32_t seed;
      int E, t[6];
      or_synth_fields(key, (uint64_t)(r * nb + c), S, k, &seed, &E, t);
      or_write_bits(out, pos, S, seed);
      or_write_bits(out, pos + (uint64_t)S, 4, (uint64_t)(E & 15));
      for (int j = 0; j < k; ++j)
        or_write_bits(out, pos + (uint64_t)(S + 4 + 4 * j), 4, (uint64_t)(t[j] & 15));
      pos += (uint64_t)or_block_bits(S, k);
    }
  }
  free(rungs);
  return pos;
}
