// Internal definitions of libseedq (sm_103a).  Not part of the C ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/seedq.h"

namespace seedq {

constexpr int kMaxJ = 9;         // hull rungs (App. B.3: four to eight on the paper's grids)
constexpr int kMaxOutliers = 16; // FP16 outlier columns (Sec. 3.5 stores four)
constexpr int kMaxBatch = 16;    // decode batch of seedq_gemm_small_batch
constexpr int kMaxCols = 65536;

// Supported rungs: S in {8,10,12,14,16}, k in {2..6} (the paper's grid, Sec. 3.1,
// at the even seed widths its Table "Rung grids" uses).
__host__ __device__ constexpr int rung_code(int S, int k) { return ((S - 8) / 2) * 5 + (k - 2); }
constexpr int kNumCodes = 25;
inline bool rung_supported(int S, int k) {
  return S >= 8 && S <= 16 && (S % 2) == 0 && k >= 2 && k <= 6;
}

#define SEEDQ_FOR_EACH_RUNG(X)                                                 \
  X(8, 2) X(8, 3) X(8, 4) X(8, 5) X(8, 6)                                      \
  X(10, 2) X(10, 3) X(10, 4) X(10, 5) X(10, 6)                                 \
  X(12, 2) X(12, 3) X(12, 4) X(12, 5) X(12, 6)                                 \
  X(14, 2) X(14, 3) X(14, 4) X(14, 5) X(14, 6)                                 \
  X(16, 2) X(16, 3) X(16, 4) X(16, 5) X(16, 6)

// Everything a kernel needs about one layer, passed by value.
struct LayerArgs {
  const uint32_t *stream;   // payload words (little-endian bit string)
  const uint64_t *row_off;  // R + 1 bit offsets
  const int32_t *brk;       // R x (J-1): first block of row r with rung > j
  const uint64_t *tables;   // nslots x 512 LFSR jump tables
  const int32_t *perm;      // C
  const uint16_t *out_vals; // R x n_out binary16
  uint32_t *flags;
  int64_t R, C;
  int32_t nb;               // C / 8 blocks per row
  int32_t J;
  int32_t L[kMaxJ];         // block bits per rung
  int32_t code[kMaxJ];      // rung_code per rung
  int32_t slot[kMaxJ];      // LFSR table slot per rung
  int32_t nslots;
  int32_t n_out;
  int32_t out_cols[kMaxOutliers];
};

}  // namespace seedq

struct seedq_layer {
  seedq::LayerArgs args;
  int32_t S[seedq::kMaxJ], k[seedq::kMaxJ];
  int32_t slot_S[seedq::kMaxJ];
  double theta[seedq::kMaxJ];
  int32_t j_tie;
  double q;
  int64_t tie_count;
  int32_t max_batch;
  uint64_t total_bits;
  int device;
  // owned device memory
  int32_t *d_perm;
  double *d_abar, *d_rho;
  float *d_rho_in, *d_a_in;
  int32_t *d_brk;
  int32_t *d_tcnt;
  uint64_t *d_row_off;
  uint64_t *d_tables;
  uint32_t *d_flags;
  uint64_t *d_summary;   // [0] total tied blocks, [1] total bits
  float *d_partials;     // split-K partial sums
  int64_t partial_elems;
  // bound stream (caller-owned)
  const void *stream;
  uint64_t stream_bytes;
};

namespace seedq {

seedq_status cuda_fail(cudaError_t e);  // records the message, returns SEEDQ_ERR_CUDA

#define SEEDQ_CUDA(call)                                                       \
  do {                                                                         \
    cudaError_t e_ = (call);                                                   \
    if (e_ != cudaSuccess) return seedq::cuda_fail(e_);                        \
  } while (0)

// ---------------------------------------------------------------- device

// Bits of the blocks of rung j within [0, x) of a row whose rung breakpoints
// are b[0..J-2] (rung j spans [b[j-1], b[j]), b[-1] = 0, b[J-1] = nb).
__device__ __forceinline__ uint64_t bits_before(const int32_t *b, int J,
                                                const int32_t *L, int nb, int x) {
  uint64_t s = 0;
  int lo = 0;
  for (int j = 0; j < J; ++j) {
    const int hi = (j < J - 1) ? b[j] : nb;
    const int cnt = min(max(x, lo), hi) - lo;
    s += (uint64_t)L[j] * (uint64_t)cnt;
    lo = hi;
  }
  return s;
}

__device__ __forceinline__ int rung_of(const int32_t *b, int J, int c) {
  int j = 0;
  for (int i = 0; i < J - 1; ++i) j += (b[i] <= c) ? 1 : 0;
  return j;
}

// 64 stream bits starting at bit `off`: lo = bits [off, off+32), hi = [off+32, off+64).
template <int NWORDS>
__device__ __forceinline__ void load_bits(const uint32_t *__restrict__ w, uint64_t off,
                                          uint32_t &lo, uint32_t &hi) {
  const uint64_t wi = off >> 5;
  const int sh = (int)(off & 31);
  const uint32_t w0 = __ldg(w + wi);
  const uint32_t w1 = __ldg(w + wi + 1);
  const uint32_t w2 = (NWORDS > 2) ? __ldg(w + wi + 2) : 0u;
  lo = __funnelshift_r(w0, w1, sh);
  hi = __funnelshift_r(w1, w2, sh);
}

template <int S, int K>
struct RungT {
  static constexpr int L = S + 4 * K + 4;
  // Words touched by a block starting at any bit offset within a word.
  static constexpr int NWORDS = (31 + L > 64) ? 3 : 2;
};

// Eq. codec for one block, exactly: I[i] = sum_j t_j (x_{iK+j} - 2^{S-1}) as an
// fp32 integer and scale = 2^(E-S+1), so w_i = I[i] * scale (exact, |I| < 2^21).
//
// The LFSR sequence prefix Q (64 bits: o_0..o_63) comes from two GF(2)-linear
// jump tables indexed by the seed's bytes (tab[v] = Q(v), tab[256+v] = Q(v<<8)).
// Each state x_n = bits [n, n+S) of Q is turned into the float 2^S + x_n by
// placing it under a fixed exponent; an FMA chain started at -1.5 * 2^S * sum t
// then yields I exactly, since every partial sum is an integer below 2^24.
template <int S, int K>
__device__ __forceinline__ void reconstruct(uint32_t lo, uint32_t hi,
                                            const uint64_t *tab, float (&I)[8],
                                            float &scale) {
  const uint64_t F = ((uint64_t)hi << 32) | lo;
  const uint32_t seed = lo & ((1u << S) - 1u);
  uint64_t Q = tab[seed & 255u];
  if (S > 8) Q ^= tab[256 + (seed >> 8)];
  const int E = ((int)(lo << (28 - S))) >> 28;  // 4-bit two's complement at bit S
  scale = __int_as_float((127 + E - S + 1) << 23);
  float tf[K];
  float T = 0.f;
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const int tj = ((int)((uint32_t)(F >> (S + 4 + 4 * j)) << 28)) >> 28;
    tf[j] = (float)tj;
    T += tf[j];
  }
  const float init = (-1.5f * (float)(1 << S)) * T;
  constexpr uint32_t EXP = (uint32_t)(127 + S) << 23;
  constexpr uint32_t MSK = ((1u << S) - 1u) << (23 - S);
  const uint32_t Qlo = (uint32_t)Q;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    float acc = init;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      const int n = i * K + j;
      const int sh = n + S - 23;
      const uint32_t w = (sh >= 0) ? (uint32_t)(Q >> (sh & 63)) : (Qlo << ((-sh) & 31));
      acc = __fmaf_rn(tf[j], __int_as_float((w & MSK) | EXP), acc);
    }
    I[i] = acc;
  }
}

__host__ __device__ inline uint64_t stream_bytes_required(uint64_t bits) {
  return ((bits + 7) / 8 + 15) / 16 * 16 + 16;
}

}  // namespace seedq
