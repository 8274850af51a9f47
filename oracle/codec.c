/*
 * Seed-Q oracle, block codec (Sec. 3.1, Eq. codec, Eq. rate).
 * TEST INFRASTRUCTURE ONLY: see seedq_oracle.h.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "seedq_oracle.h"

/* Eq. rate with m = e = 4 (Sec. 3.1: SeedLM's coefficient format is kept). */
int or_block_bits(int S, int k) { return S + 4 * k + 4; }

/* Fibonacci form over the output sequence (reading R1):
 * o_{t+S} = XOR_{i in T} o_{t+i}, seeded with the S bits of the start state. */
void or_lfsr_bits(int S, uint32_t taps, uint32_t seed, int nbits, uint8_t *o) {
  for (int t = 0; t < nbits; ++t) {
    if (t < S) {
      o[t] = (uint8_t)((seed >> t) & 1u);
    } else {
      uint8_t v = 0;
      for (int i = 0; i < S; ++i)
        if ((taps >> i) & 1u) v ^= o[t - S + i];
      o[t] = v;
    }
  }
}

/* Window state x_n = sum_{i<S} o_{n+i} 2^i; one clock shifts the window by one
 * sequence bit.  Counts clocks until state 1 comes back. */
int64_t or_lfsr_period(int S, uint32_t taps) {
  const uint32_t mask = (S == 32) ? 0xffffffffu : ((1u << S) - 1u);
  uint32_t x = 1u;
  for (int64_t n = 1; n <= ((int64_t)1 << S); ++n) {
    uint32_t fb = 0;
    for (int i = 0; i < S; ++i)
      if ((taps >> i) & 1u) fb ^= (x >> i) & 1u;
    x = ((x >> 1) | (fb << (S - 1))) & mask;
    if (x == 1u) return n;
  }
  return 0;
}

static int popcount32(uint32_t v) {
  int c = 0;
  while (v) { c += (int)(v & 1u); v >>= 1; }
  return c;
}

/* Reading R1: smallest largest tap, then fewest taps, then smallest mask.
 * A primitive polynomial has an odd number of terms, so |T| is even. */
uint32_t or_find_taps(int S) {
  const int64_t full = ((int64_t)1 << S) - 1;
  for (int m = 1; m < S; ++m) {
    for (int pc = 2; pc <= m + 1; pc += 2) {
      for (uint32_t mid = 0; mid < (1u << (m > 1 ? m - 1 : 0)); ++mid) {
        uint32_t taps = 1u | (1u << m) | (mid << 1);
        if (m == 1 && mid) continue;
        if (popcount32(taps) != pc) continue;
        if (or_lfsr_period(S, taps) == full) return taps;
      }
    }
  }
  return 0;
}

/* Eq. codec: w = U(s) t_hat with t_hat_j = t_j 2^E (one shared exponent) and
 * U_ij = (x_{ik+j} - 2^{S-1}) / 2^{S-1} in [-1, 1] (readings R2, R3). */
void or_reconstruct_block(int S, int k, uint32_t taps, uint32_t seed, int E,
                          const int *t, float w[8]) {
  uint8_t o[128];
  const int nbits = S + 8 * k - 1;
  or_lfsr_bits(S, taps, seed, nbits, o);
  const double half = ldexp(1.0, S - 1);
  for (int i = 0; i < 8; ++i) {
    double acc = 0.0;
    for (int j = 0; j < k; ++j) {
      const int n = i * k + j;
      uint32_t x = 0;
      for (int b = 0; b < S; ++b) x |= (uint32_t)o[n + b] << b;
      const double u = ((double)x - half) / half;
      acc = acc + u * (double)t[j];
    }
    w[i] = (float)ldexp(acc, E);
  }
}

uint64_t or_read_bits(const uint8_t *stream, uint64_t pos, int n) {
  uint64_t v = 0;
  for (int q = 0; q < n; ++q) {
    const uint64_t p = pos + (uint64_t)q;
    v |= (uint64_t)((stream[p >> 3] >> (p & 7)) & 1u) << q;
  }
  return v;
}

void or_write_bits(uint8_t *stream, uint64_t pos, int n, uint64_t value) {
  for (int q = 0; q < n; ++q) {
    const uint64_t p = pos + (uint64_t)q;
    const uint8_t bit = (uint8_t)(1u << (p & 7));
    if ((value >> q) & 1u) stream[p >> 3] |= bit;
    else stream[p >> 3] &= (uint8_t)~bit;
  }
}

uint64_t or_splitmix64_at(uint64_t key, uint64_t i) {
  uint64_t z = key + (i + 1u) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

void or_synth_fields(uint64_t key, uint64_t b, int S, int k, uint32_t *seed,
                     int *E, int *t) {
  const uint64_t h = or_splitmix64_at(key, b);
  const uint32_t period = (1u << S) - 1u;
  *seed = 1u + (uint32_t)(h >> 32) % period;
  *E = -8 + (int)(((h >> 24) & 255u) % 6u);
  for (int j = 0; j < k; ++j) t[j] = (int)((h >> (4 * j)) & 15u) - 8;
}

/* Solve the k x k system A x = b by Gaussian elimination with partial
 * pivoting; returns -1 when a pivot vanishes. */
static int solve_small(int k, double A[6][6], double b[6], double x[6]) {
  for (int c = 0; c < k; ++c) {
    int p = c;
    for (int r = c + 1; r < k; ++r)
      if (fabs(A[r][c]) > fabs(A[p][c])) p = r;
    if (fabs(A[p][c]) < 1e-12) return -1;
    if (p != c) {
      for (int q = 0; q < k; ++q) { double tmp = A[c][q]; A[c][q] = A[p][q]; A[p][q] = tmp; }
      double tmp = b[c]; b[c] = b[p]; b[p] = tmp;
    }
    for (int r = c + 1; r < k; ++r) {
      const double f = A[r][c] / A[c][c];
      for (int q = c; q < k; ++q) A[r][q] = A[r][q] - f * A[c][q];
      b[r] = b[r] - f * b[c];
    }
  }
  for (int r = k - 1; r >= 0; --r) {
    double s = b[r];
    for (int q = r + 1; q < k; ++q) s = s - A[r][q] * x[q];
    x[r] = s / A[r][r];
  }
  return 0;
}

/* Sec. 3.1: the encoder searches all 2^S - 1 seeds; the least-squares
 * coefficients are quantized to 4-bit mantissas under one 4-bit exponent. */
double or_encode_block(int S, int k, uint32_t taps, const double w[8],
                       uint32_t *best_seed, int *best_E, int *best_t) {
  double best = INFINITY;
  uint8_t o[128];
  const double half = ldexp(1.0, S - 1);
  for (uint32_t s = 1; s < (1u << S); ++s) {
    or_lfsr_bits(S, taps, s, S + 8 * k - 1, o);
    double U[8][6];
    for (int i = 0; i < 8; ++i)
      for (int j = 0; j < k; ++j) {
        uint32_t x = 0;
        for (int b = 0; b < S; ++b) x |= (uint32_t)o[i * k + j + b] << b;
        U[i][j] = ((double)x - half) / half;
      }
    double A[6][6], rhs[6], tstar[6];
    for (int p = 0; p < k; ++p) {
      rhs[p] = 0.0;
      for (int i = 0; i < 8; ++i) rhs[p] = rhs[p] + U[i][p] * w[i];
      for (int q = 0; q < k; ++q) {
        A[p][q] = 0.0;
        for (int i = 0; i < 8; ++i) A[p][q] = A[p][q] + U[i][p] * U[i][q];
      }
    }
    if (solve_small(k, A, rhs, tstar) != 0) continue;
    int E = -8;
    for (; E < 7; ++E) {
      int fits = 1;
      for (int j = 0; j < k; ++j) {
        const double m = nearbyint(ldexp(tstar[j], -E));
        if (m < -8.0 || m > 7.0) { fits = 0; break; }
      }
      if (fits) break;
    }
    int t[6];
    for (int j = 0; j < k; ++j) {
      double m = nearbyint(ldexp(tstar[j], -E));
      if (m < -8.0) m = -8.0;
      if (m > 7.0) m = 7.0;
      t[j] = (int)m;
    }
    double err = 0.0;
    for (int i = 0; i < 8; ++i) {
      double r = 0.0;
      for (int j = 0; j < k; ++j) r = r + U[i][j] * (double)t[j];
      const double d = w[i] - ldexp(r, E);
      err = err + d * d;
    }
    if (err < best) {
      best = err;
      *best_seed = s;
      *best_E = E;
      for (int j = 0; j < k; ++j) best_t[j] = t[j];
    }
  }
  return best;
}
