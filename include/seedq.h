/*
 * seedq.h -- C ABI of libseedq.so, a GB300 (sm_103a) implementation of the
 * inference hot path of Seed-Q ("Security-Enhanced Seed-Based Weight
 * Quantization for Large Language Models", arxiv 2609.38477): weight blocks
 * regenerated from LFSR seeds and 4-bit coefficients (Sec. 3.1, Eq. codec)
 * under the side-information-free rung schedule (Sec. 3.3-3.6, Alg. 2),
 * consumed straight away by a decode-batch matrix-vector product.
 *
 * General rules for every entry point:
 *  - Pointers marked "device" must point to memory of the current CUDA
 *    device; pointers marked "host" to ordinary host memory.  The caller owns
 *    every buffer it passes (stream, x, y, W, outlier values) and the CUDA
 *    stream.  A seedq_layer owns only the plan derived from its descriptor.
 *  - `cuda_stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Hot calls (decode, gemv, gemm) only enqueue work on it: they
 *    allocate nothing, do not synchronize, and return before the work ends.
 *  - Argument errors are reported synchronously, before any launch, and leave
 *    nothing enqueued.  SEEDQ_ERR_CUDA means a CUDA call failed; the message
 *    of the last failure is available from seedq_last_cuda_error_string().
 *  - A layer may be used from several host threads only if calls on it are
 *    serialized; different layers are independent.
 *
 * Stream format (Sec. 3.1 Eq. rate, Sec. 3.6; the paper leaves the bit order
 * open and this library fixes it): one little-endian bit string, bit p in
 * byte p>>3 at bit p&7; a block of rung (S,k) is l = S + 4k + 4 bits, fields
 * LSB first in the order seed (S bits), shared exponent E (4-bit two's
 * complement), mantissas t_0..t_{k-1} (4-bit two's complement each); blocks in
 * row-major order of the column-permuted matrix, no padding between rows.
 * The LFSR of width S is the window form o_{t+S} = XOR_{i in T_S} o_{t+i}
 * seeded with the seed's bits (see seedq_lfsr_taps), and entry (i,j) of U(s)
 * is (x_{ik+j} - 2^{S-1}) / 2^{S-1}, x_n the S-bit window after n clocks.
 */
#ifndef SEEDQ_H
#define SEEDQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SEEDQ_OK = 0,
  SEEDQ_ERR_INVALID_ARG = 1,  /* NULL pointer, bad size, non-finite factor */
  SEEDQ_ERR_STREAM = 2,       /* stream length or buffer size disagrees with the plan */
  SEEDQ_ERR_SCHEDULE = 3,     /* thresholds not increasing, tie count > tied blocks */
  SEEDQ_ERR_CUDA = 4,         /* a CUDA runtime call failed */
  SEEDQ_ERR_NOMEM = 5,        /* device or host allocation failed (prepare only) */
  SEEDQ_ERR_UNSUPPORTED = 6,  /* rung or shape outside what the kernels implement */
  SEEDQ_ERR_IO = 7,           /* a container file could not be opened, read or written */
  SEEDQ_ERR_FORMAT = 8        /* a container file is malformed, truncated or corrupted */
} seedq_status;

/* A rung g = (S, k) of the hull: seed width S and coefficient count k (Sec. 3.1).
 * Supported: S in {8, 10, 12, 14, 16}, k in {2, ..., 6}. */
typedef struct {
  int32_t S;
  int32_t k;
} seedq_rung;

/* The global decoder table of Sec. 3.6 / Alg. 2 (Require line): hull rungs,
 * thresholds and floor.  All arrays are host memory, read during prepare only.
 *   J      number of hull rungs, 1..9, rates strictly increasing.
 *   theta  J-1 thresholds, strictly increasing: theta[j] = lambda / s_j of
 *          Eq. ladder, stored as the encoder computed it (the decoder does not
 *          divide, so encoder and decoder compare the same doubles).
 *   j_tie  index of the threshold whose tied group is partially demoted
 *          (App. A.5), or -1.
 *   q      importance floor of Sec. 3.3 (imp <- max(imp, q)). */
typedef struct {
  int32_t J;
  const seedq_rung *rungs;
  const double *theta;
  int32_t j_tie;
  double q;
} seedq_schedule;

/* One weight tensor W (R x C) and the per-tensor inputs of Alg. 2.
 *   rows, cols    R, C; C a multiple of 8, 8 <= C <= 65536; 1 <= R <= 2^24.
 *   a             host, C floats, finite and >= 0, not all zero: the input
 *                 second moments (Eq. gamma or Eq. prop).
 *   rho           host, R floats finite and > 0, or NULL for all ones
 *                 (the output-side factor of Sec. 3.3).
 *   tie_count     T_t of Alg. 2: the first T_t tied blocks in row-major order
 *                 take the lower rung.
 *   n_outliers    0..16 FP16 outlier columns (Sec. 3.5, App. A.6).
 *   outlier_cols  host, n_outliers distinct column indices in [0, C).
 *   outlier_vals  device, R x n_outliers binary16 values, row-major; read by
 *                 every decode/gemv call, so it must outlive the layer.
 *   max_batch     largest n passed to seedq_gemm_small_batch (1..16); 0 = 16. */
typedef struct {
  int64_t rows;
  int64_t cols;
  const float *a;
  const float *rho;
  int64_t tie_count;
  int32_t n_outliers;
  const int32_t *outlier_cols;
  const uint16_t *outlier_vals;
  int32_t max_batch;
} seedq_layer_desc;

typedef struct seedq_layer seedq_layer;

/* Build the decoder plan of one tensor (Alg. 2 lines computing imp, the floor
 * and the ladder; App. A.7 on encoder/decoder agreement): column permutation (stable ascending
 * sort of a), unit-mean block means and row factors in fp64 in a fixed order,
 * per-row rung breakpoints after the tie pass, per-row bit offsets.  Runs on
 * the device on `cuda_stream` and waits for it (one-time set-up).  Allocates
 * the plan's device memory; *out receives the layer.  Errors: INVALID_ARG,
 * UNSUPPORTED (rung or size), SCHEDULE (theta not increasing, j_tie out of
 * range, tie_count larger than the tied group), NOMEM, CUDA. */
seedq_status seedq_layer_prepare(const seedq_layer_desc *desc,
                                 const seedq_schedule *sched, void *cuda_stream,
                                 seedq_layer **out);

/* Total payload bits the plan expects for the tensor (sum of l(g_b)). */
seedq_status seedq_layer_stream_bits(const seedq_layer *layer, uint64_t *bits);

/* Bytes a stream buffer of `bits` payload bits must span: the payload rounded
 * up to 16 bytes plus a 16-byte guard that the kernels may read (never use). */
uint64_t seedq_stream_bytes_required(uint64_t bits);

/* Attach the compressed stream (device, caller-owned, 16-byte aligned) to the
 * layer.  stream_bits must equal seedq_layer_stream_bits and stream_bytes must
 * be at least seedq_stream_bytes_required(stream_bits); otherwise
 * SEEDQ_ERR_STREAM.  The buffer must stay valid while the layer is used. */
seedq_status seedq_layer_bind_stream(seedq_layer *layer, const void *stream,
                                     uint64_t stream_bits, uint64_t stream_bytes);

/* Diagnostics: lower the number of bound-stream bytes the layer's kernels may
 * read to `bytes` (at most the bound size; it cannot be raised again without
 * binding anew).  With fewer bytes than seedq_stream_bytes_required(bits) the
 * kernels cut their reads off at the limit and set bit 0 of the device error
 * flags; the results are then wrong for the rows that reach the limit.  Used to
 * test the error flag without any out-of-bounds access.  No paper counterpart.
 * Errors: INVALID_ARG (NULL layer, bytes above the bound size), STREAM
 * (unbound). */
seedq_status seedq_layer_limit_stream_bytes(seedq_layer *layer, uint64_t bytes);

/* Free the plan (waits for the device).  NULL is accepted. */
seedq_status seedq_layer_release(seedq_layer *layer);

/* Alg. 2 in full: every block reconstructed by Eq. codec, written through the
 * inverse column permutation, outlier columns overwritten (Alg. 2 last lines).
 * W: device, R x C float32, row-major, original column order.  Values are
 * exact (each weight is I * 2^(E-S+1) with |I| < 2^21).  Needs a bound stream. */
seedq_status seedq_decode_weights(const seedq_layer *layer, float *W,
                                  void *cuda_stream);

/* Rows [row0, row0 + nrows) only; W: device, nrows x C. */
seedq_status seedq_decode_rows(const seedq_layer *layer, int64_t row0,
                               int64_t nrows, float *W, void *cuda_stream);

/* y = W_hat x (the matrix-vector product the reconstructed weights feed,
 * Sec. 1 and App. C; W_hat is never materialized).  x: device, C bfloat16
 * values (bit patterns) in the original column order; y: device, R float32.
 * Accumulation in fp32.  Errors: INVALID_ARG (NULL layer, x or y), STREAM (no
 * stream bound), CUDA (launch failed). */
seedq_status seedq_gemv(const seedq_layer *layer, const uint16_t *x, float *y,
                        void *cuda_stream);

/* Y = X W_hat^T for n = 1..max_batch activation columns: X device n x C
 * bfloat16 row-major, Y device n x R float32 row-major (row b of Y is
 * W_hat x_b).  Each block is reconstructed once and used for all n columns.
 * Errors: INVALID_ARG (NULL pointer, n outside 1..max_batch), STREAM (no
 * stream bound), CUDA. */
seedq_status seedq_gemm_small_batch(const seedq_layer *layer, const uint16_t *X,
                                    int32_t n, float *Y, void *cuda_stream);

/* Several tensors in one launch (Alg. 2 decodes each tensor on its own, in
 * no fixed order, so the tensors of a decode step are independent): for i < count,
 * Y[i] = X[i] W_hat_i^T with X[i] device n x C_i bfloat16 and Y[i] device
 * n x R_i float32, as seedq_gemm_small_batch does for one layer.  count is
 * 1..8 and every layer must be bound and allow batch n.  Work is split across
 * the SMs by the modeled cost of all tensors together.  The fused calls
 * (gemv, gemm_small_batch, gemm_multi) use per-layer scratch (permuted
 * activations, partial sums of row groups cut between SMs), so calls that
 * involve the same layer must not run concurrently on different CUDA
 * streams.  Errors: INVALID_ARG (count outside 1..8, a NULL layer, X[i] or
 * Y[i], n above some layer's max_batch), STREAM (a layer without a bound
 * stream), CUDA. */
seedq_status seedq_gemm_multi(const seedq_layer *const *layers, int32_t count,
                              const uint16_t *const *X, int32_t n, float *const *Y,
                              void *cuda_stream);

/* ------------------------------------------------------------ layer sets
 * All tensors of a model (or any group of prepared, bound layers) behind one
 * launch per call: the per-tensor descriptors and, for every batch size up to
 * the set's max_batch, the cost-balanced split of all their blocks across the
 * SMs are built once, in device memory, by seedq_layer_set_create
 * (synchronous; allocates).  A call then needs no host-side work per tensor.
 * Activations and outputs live in one buffer each: tensor i reads its
 * n x C_i bfloat16 block at X + n * col_offsets[i] and writes its n x R_i
 * float32 block at Y + n * row_offsets[i] (offsets from
 * seedq_layer_set_layout; col_offsets[count] = sum of C_i, likewise rows).
 * The set captures each layer's bound stream when it is created: rebinding or
 * releasing a layer requires releasing the set first.  Calls on a set use the
 * layers' scratch, so they must not overlap with other calls on those layers. */
typedef struct seedq_layer_set seedq_layer_set;

/* count: 1..65535 layers, each bound; max_batch of the set = the smallest.
 * Errors: INVALID_ARG (NULL array or entry, count out of range), STREAM (a
 * layer without a bound stream), NOMEM, CUDA. */
seedq_status seedq_layer_set_create(const seedq_layer *const *layers, int32_t count,
                                    seedq_layer_set **out);
/* Host arrays of count + 1 entries each (either may be NULL).  Errors:
 * INVALID_ARG (NULL set). */
seedq_status seedq_layer_set_layout(const seedq_layer_set *set, int64_t *col_offsets,
                                    int64_t *row_offsets);
/* Y_i = X_i W_hat_i^T for every tensor of the set, n = 1..max_batch (the
 * tensors are independent, Alg. 2; any order, Sec. 3.6).  Asynchronous like
 * the other hot calls.  Errors: INVALID_ARG (NULL set, X or Y, n out of
 * range), CUDA. */
seedq_status seedq_gemm_set(const seedq_layer_set *set, const uint16_t *X, int32_t n, float *Y,
                            void *cuda_stream);
seedq_status seedq_layer_set_release(seedq_layer_set *set);

/* Introspection for parity tests (the plan of Alg. 2 as the kernels hold it).
 * Host copy of the rung index (0..J-1) of blocks of rows [row0, row0+nrows):
 * rungs_host receives nrows x (C/8) bytes.  Synchronous.  Errors:
 * INVALID_ARG (NULL pointer, rows out of range), NOMEM, CUDA. */
seedq_status seedq_layer_rung_map(const seedq_layer *layer, int64_t row0,
                                  int64_t nrows, uint8_t *rungs_host);

/* Host copy of the column permutation (C int32, Sec. 3.3): block c of a row
 * holds original columns perm[8c .. 8c+7].  Synchronous.  Errors: INVALID_ARG
 * (NULL pointer), CUDA. */
seedq_status seedq_layer_perm(const seedq_layer *layer, int32_t *perm_host);

/* Host copy of the per-row bit offsets (R+1 uint64, offsets[R] = total).
 * Synchronous.  Errors: INVALID_ARG (NULL pointer), CUDA. */
seedq_status seedq_layer_row_offsets(const seedq_layer *layer, uint64_t *offsets_host);

/* Device error flags accumulated by the layer's kernels since prepare.  Bit 0:
 * the plan and the bound buffer disagree -- a kernel's read range reached past
 * the readable bytes of the stream (the read is cut off there, the affected
 * weights or rows are wrong, nothing outside the buffer is read), or the bits a
 * row's blocks occupy by its rung breakpoints differ from its row offsets.
 * Never set for a stream bound with seedq_layer_bind_stream and a plan from
 * seedq_layer_prepare.  Synchronous; 0 means no fault was seen. */
seedq_status seedq_last_device_error(const seedq_layer *layer, uint32_t *flags);

/* Tap mask T_S of the width-S LFSR used by the stream format (bit i set when
 * o_{t+i} feeds o_{t+S}); 0 for widths outside 8..16.  Host function. */
uint32_t seedq_lfsr_taps(int32_t S);

/* ---------------------------------------------------------------- encoder
 * The exhaustive seed search of Eq. codec (Sec. 3.1: every seed of the S-bit
 * LFSR, least-squares coefficients quantized to 4-bit mantissas under one
 * 4-bit exponent, smallest quantized error), run per block at its rung as
 * Alg. 1's emit step does, and the packing of the chosen fields into the
 * stream layout above.  Per seed: U(s) as in Eq. codec; the k x k normal
 * equations solved in fp64 by Gaussian elimination with partial pivoting
 * (seeds with a pivot below 1e-12 are skipped); E = the smallest value in
 * [-8, 7] for which every round-half-even t*_j 2^-E lies in [-8, 7] (7 if
 * none); t_j those values clamped to [-8, 7]; error = sum_i (w_i - w_hat_i)^2
 * in fp64.  The smallest error wins, ties to the smaller seed.  Every product
 * and sum is rounded separately in a fixed order, so the choice is the same
 * on any IEEE machine running these steps.
 *
 * Outputs per block b: seed[b] (uint32), E[b] (int8), t[6 b + j] (int8, j < k;
 * the rest 0), err[b] (double; may be NULL).  All device pointers; work is
 * enqueued on cuda_stream. */

/* Blocks at one rung (S even in 8..16, k in 2..6): w is device nblocks x 8
 * float32, row-major (one block per row).  Other rungs: SEEDQ_ERR_UNSUPPORTED. */
seedq_status seedq_encode_blocks(int32_t S, int32_t k, const float *w, int64_t nblocks,
                                 uint32_t *seed, int8_t *E, int8_t *t, double *err,
                                 void *cuda_stream);

/* Every block of a prepared layer at the rung its plan assigns: W is device
 * R x C float32 in the original column order (block (r, c) holds the columns
 * perm[8c .. 8c+7] of row r); outputs have R x (C/8) entries in row-major
 * block order.  The layer's outlier columns enter the search as zero: their
 * FP16 values overwrite the decoded columns (Sec. 3.5), and a spike left in
 * place would distort its seven block-mates. */
seedq_status seedq_encode_layer(const seedq_layer *layer, const float *W, uint32_t *seed,
                                int8_t *E, int8_t *t, double *err, void *cuda_stream);

/* Pack per-block fields (as seedq_encode_layer writes them) into a stream
 * buffer: device, 16-byte aligned, stream_bytes >= seedq_stream_bytes_required
 * (plan bits); zeroed first.  The result binds to the layer with
 * seedq_layer_bind_stream. */
seedq_status seedq_pack_stream(const seedq_layer *layer, const uint32_t *seed, const int8_t *E,
                               const int8_t *t, void *stream, uint64_t stream_bytes,
                               void *cuda_stream);

/* Measurement helper for the encoder's roofline (no paper counterpart): one
 * launch of blocks_per_sm x SMs CTAs of 256 threads, each thread running eight
 * independent fp64 FMA chains for `iters` steps, so the device's fp64 FMA
 * pipe bounds it.  *fmas receives the FMAs the launch performs (2 flops each);
 * the caller times it on cuda_stream.  out: device, one double (written only
 * in a case that does not arise; it keeps the chains from being removed).
 * Asynchronous.  Errors: INVALID_ARG (iters < 1, blocks_per_sm outside 1..64,
 * NULL pointer), CUDA. */
seedq_status seedq_fp64_fma_probe(int64_t iters, int32_t blocks_per_sm, double *out,
                                  void *cuda_stream, int64_t *fmas);

/* -------------------------------------------------------------- container
 * A file holding a compressed model: the global decoder table (Sec. 3.6, as
 * seedq_schedule) and, per tensor, what Alg. 2 reads besides it: shape,
 * importance factors a and rho (the decoder recomputes the rung map from
 * them), T_t, the FP16 outlier columns (Sec. 3.5) and the payload stream.
 * Little-endian, no padding; the header records the LFSR taps of S = 8..16
 * (a file written with other taps is rejected with SEEDQ_ERR_UNSUPPORTED) and
 * the file ends in a 64-bit FNV-1a hash of its contents (checked on open).
 * Host functions; they never touch the GPU.
 *
 * Per-tensor view.  All pointers are host memory: on write they are read
 * only; from seedq_container_get they point into the container and stay valid
 * until seedq_container_close.  outlier_vals is rows x n_outliers binary16
 * (host here, unlike seedq_layer_desc, which wants them on the device);
 * stream holds ceil(stream_bits / 8) bytes. */
typedef struct {
  const char *name;
  int64_t rows;
  int64_t cols;
  const float *a;
  const float *rho;           /* NULL: all ones */
  int64_t tie_count;
  int32_t n_outliers;
  const int32_t *outlier_cols;
  const uint16_t *outlier_vals;
  const uint8_t *stream;
  uint64_t stream_bits;
} seedq_container_tensor;

typedef struct seedq_container seedq_container;

/* Write the schedule and ntensors tensors to path (replacing the file).
 * Errors: INVALID_ARG (NULL or inconsistent schedule or tensor fields), IO. */
seedq_status seedq_container_write(const char *path, const seedq_schedule *sched,
                                   int32_t ntensors, const seedq_container_tensor *tensors);
/* Read and validate a container; *out receives it (release with _close).
 * Errors: IO, FORMAT (bad magic, version, sizes, hash), UNSUPPORTED (taps). */
seedq_status seedq_container_open(const char *path, seedq_container **out);
/* The stored schedule; its arrays point into the container. */
seedq_status seedq_container_schedule(const seedq_container *c, seedq_schedule *sched);
seedq_status seedq_container_count(const seedq_container *c, int32_t *ntensors);
seedq_status seedq_container_get(const seedq_container *c, int32_t index,
                                 seedq_container_tensor *tensor);
seedq_status seedq_container_close(seedq_container *c);

/* Fill a stream buffer with the synthetic payload of the workload recipe:
 * block b of the tensor (row-major) draws h = splitmix64 output number b from
 * state `key` and uses seed = 1 + (h>>32) mod (2^S-1), E = -8 + ((h>>24)&255)
 * mod 6, t_j = ((h>>4j)&15) - 8 at the rung the plan assigns.  stream: device,
 * stream_bytes >= seedq_stream_bytes_required(plan bits); zeroed first.  A
 * benchmark and test input generator, not part of the paper's method.
 * Synchronous.  Errors: INVALID_ARG (NULL layer or stream, stream not 16-byte
 * aligned), STREAM (buffer too small), CUDA. */
seedq_status seedq_synth_stream(const seedq_layer *layer, uint64_t key,
                                void *stream, uint64_t stream_bytes,
                                void *cuda_stream);

/* Allocation-free per-row schedule pass, for callers that cannot call
 * cudaMalloc when they need it (a fixed memory budget reserved up front, an
 * allocator-less runtime, code that must not touch the CUDA allocator while
 * other work is in flight).  The paper has no counterpart: it is the row part
 * of seedq_layer_prepare (per-row rung breakpoints, the tie pass, row bit
 * offsets) run on caller buffers, with its temporary per-row tie counts in a
 * file-scope device array of SEEDQ_STATIC_PLAN_MAX_ROWS entries (512 KiB held
 * by every GPU that loads the library until exit).  It allocates nothing.
 *   abar      device, nb doubles: unit-mean block means of the permuted a.
 *   rho       device, rows doubles: unit-mean row factors (all 1 if none).
 *   rows, nb  R (1..SEEDQ_STATIC_PLAN_MAX_ROWS) and C/8; larger R returns
 *             SEEDQ_ERR_UNSUPPORTED.
 *   brk       device, rows x (J-1) int32 out: first block of each row with
 *             rung > j (may be NULL when J == 1).
 *   row_off   device, rows + 1 uint64 out (row_off[rows] = total bits).
 *   summary   device, 2 uint64 out: tied blocks at theta[j_tie], total bits;
 *             the caller checks tie_count <= summary[0].
 * Every call looks up the array's device address with the current device; the
 * first call on a device also loads the library's module there, so make it
 * before any stream capture.  The rung lengths travel in the kernel
 * parameters, so the call makes no host-to-device copy.  Work is enqueued on
 * cuda_stream and not waited for.  Calls share the array: calls that overlap
 * on the GPU (other streams, other threads) race and must be serialized. */
#define SEEDQ_STATIC_PLAN_MAX_ROWS (1 << 17)
seedq_status seedq_row_plan_static(const double *abar, const double *rho, int64_t rows,
                                   int32_t nb, const seedq_schedule *sched,
                                   int64_t tie_count, int32_t *brk, uint64_t *row_off,
                                   uint64_t *summary, void *cuda_stream);

/* ------------------------------------------- data-free importance (Sec. 3.2)
 * What the encoder computes from an FP16 checkpoint before allocating rungs:
 * the input-side factor a of every tensor, the output-side factor rho of the
 * rows that write the residual stream, and the outlier columns (Sec. 3.5).
 *
 *   Eq. gamma: a = gamma^2 for q, k, v (gain of the attention input norm),
 *     gate, up (gain of the MLP input norm) and the head (final norm).
 *   Eq. prop:  a^(o) = repeat_kv((W_v o W_v) a^(in)) (query head h reads
 *     key-value head h / (n_heads / n_kv_heads)); a^(down)_c = E[silu(g)^2]
 *     ((W_up o W_up) a^(in))_c, g ~ N(0, ((W_gate o W_gate) a^(in))_c), the
 *     expectation by 64-node Gauss-Hermite quadrature.
 *   Backward proxy (Sec. 3.2 output side, App. A.1): G = (W_head o W_head)^T 1;
 *     for each layer, last first: rho_down = G; G += (W_gate o W_gate)^T Gh +
 *     (W_up o W_up)^T Gh with Gh = (W_down o W_down)^T G; rho_o = G;
 *     G += (W_v o W_v)^T Gv with Gv the sum over the query heads of each
 *     key-value head of (W_o o W_o)^T G.  Norms are the identity here; rows of
 *     q, k, v, gate, up and the head have rho = 1.  The stored rho vectors
 *     are divided by their mean (summed in row order): the proxy's overall
 *     scale grows by a model-dependent factor per layer and carries no
 *     information (the plan normalizes both factors to unit mean anyway).
 *   Outlier statistics (Sec. 3.5, App. A.6): per column of every tensor the
 *     dynamic range max_i |W_ij| / (median_i |W_ij| + 2^-24) (the median of an
 *     even count is the mean of the two middle values) and the activation
 *     ratio a_j / mean(a) (mean summed in column order).
 *
 * Weights are FP16 bit patterns, row-major [out][in] (rows = outputs), every
 * matrix 16-byte aligned with in-dimension a multiple of 32; gains FP16 too.
 * All weight and table pointers are device pointers. */
typedef struct {
  const uint16_t *attn_norm, *mlp_norm;  /* d_model gains */
  const uint16_t *wq, *wk, *wv, *wo, *wgate, *wup, *wdown;
} seedq_llama_layer;

typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ff;
  int64_t vocab;
  const seedq_llama_layer *layers; /* host array of n_layers entries */
  const uint16_t *final_norm;      /* d_model gain of the head's input */
  const uint16_t *lm_head;         /* vocab x d_model */
} seedq_llama_model;

/* Outputs.  Tensor order of the model: per layer q, k, v, o, gate, up, down,
 * then the head; "columns in model order" concatenates every tensor's in-
 * dimension in that order. */
typedef struct {
  float *a_o;        /* n_layers x (n_heads head_dim), float32 (App. A.7)     */
  float *a_down;     /* n_layers x d_ff                                       */
  float *rho_o;      /* n_layers x d_model: rho of W_o's rows, unit mean      */
  float *rho_down;   /* n_layers x d_model: rho of W_down's rows, unit mean   */
  double *dyn_range; /* optional: columns in model order; the statistic where
                        it is >= 1e3, else 0                                 */
  double *act_ratio; /* optional: columns in model order                      */
} seedq_importance_out;

/* One stored outlier column: tensor index in model order and column. */
typedef struct {
  int32_t tensor, column;
} seedq_outlier;

/* The whole analysis over a resident model: tables into *out, then the
 * outlier selection of App. A.6 (each rule's candidates, dynamic range >= 1e3
 * and activation ratio >= 1e2, at most 32 per rule by decreasing statistic,
 * ties by tensor then column; ranked by the better position in the two lists,
 * ties by tensor then column) into outliers[0..*n_outliers), at most
 * max_outliers (the paper stores four).  Synchronous: enqueues on cuda_stream,
 * waits for it, and allocates and frees device scratch.  Errors:
 * SEEDQ_ERR_INVALID_ARG (null or misaligned pointers, shapes out of range,
 * in-dimension not a multiple of 32, n_heads not a multiple of n_kv_heads),
 * SEEDQ_ERR_NOMEM, SEEDQ_ERR_CUDA. */
seedq_status seedq_importance(const seedq_llama_model *model, const seedq_importance_out *out,
                              seedq_outlier *outliers, int32_t max_outliers,
                              int32_t *n_outliers, void *cuda_stream);

/* Outlier statistics of one matrix (the column pass of seedq_importance
 * alone): dyn_range as above for its C columns (device, C doubles), and the
 * column sums of squares weighted by row, col_sq[c] = sum_r W_rc^2 g_r (device,
 * C doubles; g device R floats, or NULL for all ones; col_sq may be NULL).
 * W device R x C FP16, 16-byte aligned, C a multiple of 32.  Enqueued, not
 * waited for. */
seedq_status seedq_column_stats(const uint16_t *W, int64_t R, int64_t C, const float *g,
                                double *dyn_range, double *col_sq, void *cuda_stream);

/* Test / benchmark input generator (no paper counterpart): n FP16 values
 * out[i] = fp16_rn(z_i m 2^-e), z_i the sum of the four 16-bit fields of
 * splitmix64 output number first + i of state key, minus 131070; m in
 * 1..63, e in 0..40 (exact in float32 before the rounding).  out device,
 * 16-byte aligned.  Enqueued, not waited for. */
seedq_status seedq_synth_fp16(uint64_t key, int64_t first, int64_t n, int32_t m, int32_t e,
                              uint16_t *out, void *cuda_stream);

/* ------------------------------------------------- allocator (Alg. 1, Sec. 3.4)
 * The encoder-side allocation over a set of tensors sharing one budget: the
 * floor q = the m-th smallest raw importance over all blocks, m =
 * ceil(floor_f N); the multiplier lambda by bisection over its IEEE bit
 * pattern so that the payload bits with thresholds theta_j = lambda / s_j meet
 * floor(8 rbar N); the tied group at the critical threshold and its demotion
 * count, spread over the tensors in tensor order (App. A.5).  Importance is
 * that of Eq. imp with the plan's fixed-order fp64 factors (App. A.7).
 *   tensors     host array of count descriptors; a and rho are HOST float32
 *               arrays (rho NULL = 1 on every row); cols a multiple of 8.
 *   J, S, k     the hull's rungs in increasing rate (S even 8..16, k 2..6).
 *   slopes      J - 1 hull slopes s_j (decreasing).
 *   theta       out, J - 1 thresholds; j_tie, q out; tie_count and
 *               stream_bits out, count entries each (payload bits per tensor).
 * Synchronous; allocates.  Errors: SEEDQ_ERR_INVALID_ARG, SEEDQ_ERR_SCHEDULE
 * (budget infeasible, or more than one tied group straddles the budget),
 * SEEDQ_ERR_NOMEM, SEEDQ_ERR_CUDA. */
typedef struct {
  int64_t rows, cols;
  const float *a;   /* host, cols */
  const float *rho; /* host, rows, or NULL */
} seedq_factor_desc;

seedq_status seedq_allocate(const seedq_factor_desc *tensors, int32_t count, int32_t J,
                            const int32_t *S, const int32_t *k, const double *slopes,
                            double rbar, double floor_f, double *theta, int32_t *j_tie,
                            double *q, int64_t *tie_count, uint64_t *stream_bits,
                            void *cuda_stream);

const char *seedq_status_string(seedq_status status);
const char *seedq_last_cuda_error_string(void);

#ifdef __cplusplus
}
#endif
#endif /* SEEDQ_H */
