/*
 * Seed-Q CPU oracle: a plain, slow, obviously-correct restatement of the
 * decoder of "Security-Enhanced Seed-Based Weight Quantization for Large
 * Language Models" (arxiv 2609.38477), plus the encoder-side pieces needed to
 * make its inputs (hull, allocator, brute-force seed search).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this library: only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark use it.  It shares no code, header, table or constant with
 * the CUDA library; the two meet only through seeded inputs.
 *
 * Floating point: fp64 everywhere, compiled with -ffp-contract=off so that
 * every product and sum is one IEEE-rounded operation in the order written.
 *
 * Conventions (readings of the paper that it leaves open are marked R#):
 *   - B = 8 weights per block, m = e = 4 (Sec. 3.1, Eq. rate).
 *   - A rung is (S, k); rung indices are 0-based here (the paper counts 1..J).
 *   - theta[j], j = 0..J-2, is the threshold for moving from rung j to j+1
 *     (Eq. ladder: lambda / s_j, stored as the encoder computed it).
 *   - Stream: one little-endian bit string, bit p in byte p>>3 at bit p&7,
 *     fields LSB first, block field order seed(S) | E(4) | t_0..t_{k-1}(4 each),
 *     blocks in row-major block order of the permuted matrix, no row padding.
 */
#ifndef SEEDQ_ORACLE_H
#define SEEDQ_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------- codec (Sec. 3.1, Eq. codec and Eq. rate) ---------------- */

/* Eq. rate: l(S,k) = S + m k + e bits with m = e = 4. */
int or_block_bits(int S, int k);

/* LFSR sequence (reading R1/R2): o_0..o_{S-1} are the seed bits, LSB first;
 * o_{t+S} = XOR over taps i of o_{t+i}, where bit i of `taps` marks tap i
 * (bit 0 must be set).  Writes nbits sequence bits into o[]. */
void or_lfsr_bits(int S, uint32_t taps, uint32_t seed, int nbits, uint8_t *o);

/* Period of the window-state sequence started at state 1 (0 if it never
 * returns within 2^S steps). */
int64_t or_lfsr_period(int S, uint32_t taps);

/* Brute-force choice of the feedback taps for width S (reading R1): among
 * primitive characteristic polynomials x^S + sum_{i in T} x^i (0 in T), the
 * one with the smallest largest tap below S, then the fewest taps, then the
 * smallest tap mask.  Primitive is tested as period 2^S - 1. */
uint32_t or_find_taps(int S);

/* Eq. codec for one block: w_i = 2^E * sum_j U_ij t_j, where
 * U_ij = (x_{ik+j} - 2^{S-1}) / 2^{S-1} and x_n is the S-bit LFSR state after
 * n clocks from the seed (readings R2, R3, R4).  Exact in fp64; the value is
 * then exactly representable in fp32. */
void or_reconstruct_block(int S, int k, uint32_t taps, uint32_t seed, int E,
                          const int *t, float w[8]);

/* Bit-field helpers on the stream (reading R4). */
uint64_t or_read_bits(const uint8_t *stream, uint64_t pos, int n);
void or_write_bits(uint8_t *stream, uint64_t pos, int n, uint64_t value);

/* ---------------- schedule (Sec. 3.3, 3.4, 3.6; Alg. 2) ---------------- */

typedef struct {
  int J;                /* number of hull rungs */
  const int *S;         /* J seed widths, rates increasing */
  const int *k;         /* J coefficient counts */
  const double *theta;  /* J-1 thresholds */
  int j_tie;            /* threshold index whose tied group is demoted, -1 none */
  double q;             /* importance floor */
} or_schedule;

/* Per-tensor factors of Eq. imp, built in the fixed fp64 order that App. A.7
 * requires for encoder/decoder agreement: perm = stable ascending sort of a
 * (Sec. 3.3, block importance); abar[c] = mean of a over block c of the permuted columns,
 * summed in i order, divided by its mean over c (summed in ascending c);
 * rho[r] = rho_r divided by its mean over r (summed in ascending r), or 1. */
typedef struct {
  int64_t R, C;
  int32_t *perm;  /* C */
  double *abar;   /* C/8 */
  double *rho;    /* R */
  int rho_uniform; /* 1 when every rho[r] == 1 (all rows share one rung map) */
} or_factors;

/* Not safe to call from two threads at once: the sort keeps its key in a
 * file-scope pointer.  The other functions only read their factors. */
int or_factors_init(or_factors *f, int64_t R, int64_t C, const float *a,
                    const float *rho /* NULL => all ones */);
void or_factors_free(or_factors *f);

/* Floored importance of block (r, c): max(abar[c] * rho[r], q). */
double or_imp(const or_factors *f, const or_schedule *s, int64_t r, int64_t c);

/* Eq. ladder without the tie pass: number of thresholds <= imp (0-based rung). */
int or_ladder(const or_schedule *s, double imp);

/* Rungs of rows [r0, r0+nrows) after the tie pass of Alg. 2: the first
 * tie_count blocks (row-major order over the whole tensor) whose importance
 * equals theta[j_tie] take the lower rung.  out is nrows x (C/8). */
void or_rung_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                  int64_t r0, int64_t nrows, uint8_t *out);

/* Demotions still to apply when row r0 starts (tie_count minus the tied
 * blocks of rows [0, r0), floored at 0). */
int64_t or_tie_remaining(const or_factors *f, const or_schedule *s,
                         int64_t tie_count, int64_t r0);

/* Rungs of rows [r0, r0+nrows) continuing from *remaining demotions. */
void or_rung_rows_cont(const or_factors *f, const or_schedule *s,
                       int64_t *remaining, int64_t r0, int64_t nrows,
                       uint8_t *out);

/* Number of blocks of the tensor whose floored importance equals theta[j_tie]. */
int64_t or_tied_blocks(const or_factors *f, const or_schedule *s);

/* Payload bits of rows [0, r) of the tensor (so or_row_bit_offset(f,s,T,R) is
 * the tensor's total stream length). */
uint64_t or_row_bit_offset(const or_factors *f, const or_schedule *s,
                           int64_t tie_count, int64_t r);

/* ---------------- decoder (Alg. 2) ---------------- */

/* Decode rows [r0, r0+nrows) into W (nrows x C, original column order):
 * parse blocks left to right from the row's bit offset, reconstruct with
 * Eq. codec, apply the inverse permutation, overwrite outlier columns with
 * their fp16 values (outlier_vals is R x n_out, row-major).
 * taps[S] gives the tap mask for width S.  Returns 0, or -1 if a block would
 * read past stream_bits. */
int or_decode_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                   const uint8_t *stream, uint64_t stream_bits,
                   const uint32_t *taps, int n_out, const int32_t *outlier_cols,
                   const uint16_t *outlier_vals, int64_t r0, int64_t nrows,
                   float *W);

/* y[r] = sum_c W[r,c] x[c] in fp64, x given as bf16 bit patterns (nb columns
 * of x, row-major nb x C; y is nb x nrows). */
void or_gemv_f64(int64_t nrows, int64_t C, const float *W, int nb,
                 const uint16_t *x_bf16, double *y);

/* Multi-threaded decode + fp64 GEMV of rows [r0, r0+nrows) (y is nb x R),
 * used to time the oracle as a CPU baseline.  Returns the thread count used,
 * or -1 if the stream is too short. */
int or_decode_gemv_threads(const or_factors *f, const or_schedule *s,
                           int64_t tie_count, const uint8_t *stream,
                           uint64_t stream_bits, const uint32_t *taps,
                           int nb, const uint16_t *x_bf16, int64_t r0,
                           int64_t nrows, double *y, int nthreads);

/* ---------------- synthetic payload (counter-based generator) ---------------- */

/* splitmix64 (Steele, Lea, Flood 2014): output number i (0-based) of the
 * generator whose state starts at `key`. */
uint64_t or_splitmix64_at(uint64_t key, uint64_t i);

/* Fields of block b of a synthetic tensor at rung (S,k): h = splitmix64_at(key, b);
 * seed = 1 + (h >> 32) mod (2^S - 1); E = -8 + ((h >> 24) & 255) mod 6;
 * t_j = ((h >> 4j) & 15) - 8. */
void or_synth_fields(uint64_t key, uint64_t b, int S, int k, uint32_t *seed,
                     int *E, int *t);

/* Pack the synthetic stream of rows [0, R) into stream (zeroed by the caller,
 * length >= ceil(bits/8)).  Returns the number of bits written. */
uint64_t or_synth_pack(const or_factors *f, const or_schedule *s,
                       int64_t tie_count, uint64_t key, uint8_t *stream);

/* Rows [r0, r0+nrows) of a synthetic tensor straight from its block fields,
 * equal to decoding the stream or_synth_pack writes (W: nrows x C). */
void or_synth_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                   uint64_t key, const uint32_t *taps, int n_out,
                   const int32_t *outlier_cols, const uint16_t *outlier_vals,
                   int64_t r0, int64_t nrows, float *W);

/* y (and, when yabs is not NULL, sum_c |W_rc| |x_c|) for rows [r0, r0+nrows)
 * of a synthetic tensor, from its fields, in fp64 over nthreads threads.
 * y and yabs are nb x R (only the requested rows are written). */
int or_synth_gemv_threads(const or_factors *f, const or_schedule *s, int64_t tie_count,
                          uint64_t key, const uint32_t *taps, int nb,
                          const uint16_t *x_bf16, int64_t r0, int64_t nrows, double *y,
                          double *yabs, int nthreads);

/* Pack rows [r0, r0+nrows) of the synthetic stream at bit 0 of out (zeroed by
 * the caller); returns the bits written. */
uint64_t or_synth_pack_rows(const or_factors *f, const or_schedule *s, int64_t tie_count,
                            uint64_t key, int64_t r0, int64_t nrows, uint8_t *out);

/* ---------------- encoder side (Sec. 3.4, App. A.5, Eq. codec search) ------ */

/* Lower convex hull of the points (rate(S_i,k_i), e_i) (Sec. 3.4; reading R10:
 * lower e kept per rate, collinear points dropped).  Writes hull indices in
 * increasing rate to idx, returns J. */
int or_hull(int n, const int *S, const int *k, const double *e, int *idx);

/* Allocator of Alg. 1 for a set of tensors sharing one budget: floor q at the
 * f-quantile of all blocks' importance, bisection on lambda for mean payload
 * rate <= rbar, then the tie pass demoting the critical tied group in block
 * order (tensor order, then row-major).  slopes has J-1 entries.  Outputs
 * theta (J-1), j_tie, q, tie_count[nt], bits[nt].  Returns 0 or -1 when the
 * budget is infeasible. */
int or_allocate(int nt, const or_factors *const *f, int J, const int *S,
                const int *k, const double *slopes, double rbar, double floor_f,
                double *theta, int *j_tie, double *q, int64_t *tie_count,
                uint64_t *bits);

/* Exhaustive seed search of Eq. codec for one block: for every seed in
 * [1, 2^S - 1], least-squares coefficients, then the smallest shared exponent
 * E in [-8, 7] whose rounded mantissas fit in [-8, 7]; keeps the smallest
 * quantized squared error (ties to the smaller seed).  Reading R17. */
double or_encode_block(int S, int k, uint32_t taps, const double w[8],
                       uint32_t *seed, int *E, int *t);

#ifdef __cplusplus
}
#endif
#endif
