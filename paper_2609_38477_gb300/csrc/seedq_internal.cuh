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
constexpr int kTableSlots = 5;   // jump tables for S = 8, 10, 12, 14, 16

// Supported rungs: S in {8,10,12,14,16}, k in {2..6} (the paper's grid, Sec. 3.1,
// at the even seed widths of its rung-grid table).
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
  const int32_t *perm;      // C: block c holds columns perm[8c..8c+7]
  const int32_t *invperm;   // C: position of column j in the permuted order
  const uint16_t *out_vals; // R x n_out binary16
  const int32_t *rowperm;   // R: order in which rows are grouped 32 to a warp
  float *xperm;             // max_batch x C: activations in permuted column order
  int32_t *counters;        // row groups: arrivals of partial sums (0 between calls)
  float *slots;             // max_ctas x 2 x 32 x 16 partial sums of row groups
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
  uint32_t zero;            // 0; see RungConsts
};

}  // namespace seedq

namespace seedq {
// Modeled time of one block pass of the fused kernel at rung k with n
// activation columns, in units of one coefficient: k + cost_block(n).  The
// constants are fitted to the kernel's measured time per block on
// single-rung tensors (S = 8..16, k = 2..6; n = 1, 4, 16; 2 and 8 between).
constexpr double kCostK = 1.0;
inline double cost_block(int n) {
  return n <= 1 ? 3.7 : n <= 2 ? 5.3 : n <= 4 ? 8.4 : n <= 8 ? 12.5 : 19.6;
}
// Stage width (blocks) the work profile assumes.
constexpr int kCostStage = 24;
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
  int32_t *d_invperm;
  double *d_abar, *d_rho;
  float *d_rho_in, *d_a_in;
  int32_t *d_brk;
  int32_t *d_tcnt;
  int32_t *d_rowperm;
  int32_t *d_counters;
  float *d_slots;
  float *d_xperm;
  int32_t max_ctas;      // CTAs of the fused kernel (one per SM)
  // Host-side work profile of the fused kernel, per row group (G + 1 entries,
  // cumulative): block passes the warp makes, and the sum of k over them.
  double *h_gp, *h_gk;
  int32_t *h_repbk;      // host: breakpoints of each row group's first row (G x (J-1))
  uint64_t *d_row_off;
  uint64_t *d_tables;
  uint32_t *d_flags;
  uint64_t *d_summary;   // [0] total tied blocks, [1] total bits
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

// ---------------------------------------------------------- reconstruction
//
// Eq. codec for one block, exactly: I[i] = sum_j t_j (x_{iK+j} - 2^{S-1}) as an
// fp32 integer and scale = 2^(E-S+1), so w_i = I[i] * scale (exact, |I| < 2^21).
//
// LFSR: the 64-bit sequence prefix Q = o_0..o_63 comes from two GF(2)-linear
// jump tables indexed by the seed's bytes: tab[v] = Q(v), tab[256+v] =
// Q((v mod 2^(S-8)) << 8), so the raw second byte of the field word indexes it.
//
// States as floats: a state x_n sits at bits [n, n+S) of Q.  One funnel shift
// brings a window of Q such that x_n lies at mantissa bits [23-S-d, 23-d) of a
// 32-bit word; masking it and OR-ing exponent 127+S+d gives the float
// 2^(S+d) + x_n.  A group of G consecutive states of one weight shares one
// window (d = 0..G-1).  An FMA chain from init = -sum_j t_j (2^(S+d_j) + 2^(S-1))
// then yields I exactly, provided every partial sum stays an integer below
// 2^24 in magnitude; group_size() picks the largest G for which the worst case
// (all |t_j| = 8) satisfies that.

__host__ __device__ constexpr long long exact_bound(int S, int K, int G) {
  long long s = 0;
  for (int j = 0; j < K; ++j) {
    const int d = (K - 1 - j) % G;
    s += 8ll * ((1ll << (S + d)) + (1ll << (S - 1)));
  }
  return s + 48ll * (1ll << (S - 1));
}

__host__ __device__ constexpr int group_size(int S, int K) {
  int g = 1;
  for (int G = 1; G <= K; ++G)
    if (exact_bound(S, K, G) < (1ll << 24) && S + G <= 24) g = G;
  return g;
}

// Window (lo, mid, hi hold bits [0,32), [16,48), [32,64) of the block's field
// word) and in-window bit position of the signed 4-bit field at absolute bit P;
// the field must lie in mantissa bits [0, 23) of its window.
__host__ __device__ constexpr int field_window(int P) { return P + 4 <= 23 ? 0 : P - 16 + 4 <= 23 ? 1 : 2; }
__host__ __device__ constexpr int field_pos(int P) { return P - 16 * field_window(P); }

// Per-rung constants kept in registers.  They are built from a runtime zero so
// the compiler cannot fold them into instruction immediates: a LOP3 takes one
// immediate at most, and (w & mask) | exponent must stay a single LOP3.
template <int S, int K>
struct RungConsts {
  static constexpr int G = group_size(S, K);
  uint32_t e_msk, e_x;           // shared exponent field
  uint32_t t_msk[K], t_x[K];     // mantissa fields t_j
  uint32_t s_msk[G], s_exp[G];   // state windows, by offset d within a group
  __device__ __forceinline__ explicit RungConsts(uint32_t z) {
    e_msk = (15u << S) ^ z;
    e_x = (8u << S) ^ z;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      const int P = field_pos(S + 4 + 4 * j);
      t_msk[j] = (15u << P) ^ z;
      t_x[j] = ((8u << P) | ((uint32_t)(150 - P) << 23)) ^ z;
    }
#pragma unroll
    for (int d = 0; d < G; ++d) {
      s_msk[d] = (((1u << S) - 1u) << (23 - S - d)) ^ z;
      s_exp[d] = ((uint32_t)(127 + S + d) << 23) ^ z;
    }
  }
};

// Single three-input logic instructions (the compiler otherwise splits them).
__device__ __forceinline__ uint32_t lop_and_xor(uint32_t a, uint32_t m, uint32_t x) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(r) : "r"(a), "r"(m), "r"(x));  // (a & m) ^ x
  return r;
}
__device__ __forceinline__ uint32_t lop_and_or(uint32_t a, uint32_t m, uint32_t x) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(a), "r"(m), "r"(x));  // (a & m) | x
  return r;
}

template <int S, int K, int J = 0>
__device__ __forceinline__ void coeffs(uint32_t lo, uint32_t mid, uint32_t hi,
                                       const RungConsts<S, K> &rc, float (&tf)[K]) {
  if constexpr (J < K) {
    constexpr int P = S + 4 + 4 * J;
    constexpr int W = field_window(P);
    constexpr int PP = field_pos(P);
    static_assert(PP >= 0 && PP + 4 <= 23, "field outside the mantissa");
    const uint32_t w = (W == 0) ? lo : (W == 1) ? mid : hi;
    // Under exponent 150-PP the field reads as 2^(23-PP) + (t ^ 8) = 2^(23-PP) + 8 + t.
    tf[J] = __uint_as_float(lop_and_xor(w, rc.t_msk[J], rc.t_x[J])) - (float)((1 << (23 - PP)) + 8);
    coeffs<S, K, J + 1>(lo, mid, hi, rc, tf);
  }
}

// 32 bits of Q (qlo | qhi << 32) starting at bit SH (SH may be negative: the
// window then begins below bit 0 and its low bits are zero).
template <int SH>
__device__ __forceinline__ uint32_t qwin(uint32_t qlo, uint32_t qhi) {
  if constexpr (SH <= -32) return 0u;
  else if constexpr (SH < 0) return qlo << (-SH);
  else if constexpr (SH == 0) return qlo;
  else if constexpr (SH < 32) return __funnelshift_r(qlo, qhi, SH);
  else if constexpr (SH == 32) return qhi;
  else return qhi >> (SH - 32);
}

template <int S, int K, int G, int I, int J>
__device__ __forceinline__ float state_chain(uint32_t qlo, uint32_t qhi, const RungConsts<S, K> &rc,
                                             const float (&tf)[K], float acc) {
  if constexpr (J < 0) {
    return acc;
  } else {
    // Group holding state J of weight I: its top state jt sits at d = 0.
    constexpr int grp = (K - 1 - J) / G;
    constexpr int jt = K - 1 - grp * G;
    constexpr int d = jt - J;
    const uint32_t win = qwin<I * K + jt + S - 23>(qlo, qhi);
    acc = __fmaf_rn(tf[J], __uint_as_float(lop_and_or(win, rc.s_msk[d], rc.s_exp[d])), acc);
    return state_chain<S, K, G, I, J - 1>(qlo, qhi, rc, tf, acc);
  }
}

template <int S, int K, int G, int I>
__device__ __forceinline__ void weights_from(uint32_t qlo, uint32_t qhi, const RungConsts<S, K> &rc,
                                             const float (&tf)[K], float init, float (&Iv)[8]) {
  if constexpr (I < 8) {
    Iv[I] = state_chain<S, K, G, I, K - 1>(qlo, qhi, rc, tf, init);
    weights_from<S, K, G, I + 1>(qlo, qhi, rc, tf, init, Iv);
  }
}

// lo, hi: the block's 64 field bits starting at its first bit.
template <int S, int K>
__device__ __forceinline__ void reconstruct(uint32_t lo, uint32_t hi, const uint64_t *tab,
                                            const RungConsts<S, K> &rc, float (&I)[8],
                                            float &scale) {
  constexpr int G = RungConsts<S, K>::G;
  static_assert(exact_bound(S, K, G) < (1ll << 24), "FMA chain would round");
  uint64_t Q = tab[lo & 255u];
  if (S > 8) Q ^= tab[256 + __byte_perm(lo, 0, 0x4441)];
  const uint32_t qlo = (uint32_t)Q, qhi = (uint32_t)(Q >> 32);
  // scale = 2^(E-S+1): (E+8) = field ^ 8 lands in the exponent via one multiply-add.
  const uint32_t e8 = lop_and_xor(lo, rc.e_msk, rc.e_x);
  scale = __uint_as_float(e8 * (1u << (23 - S)) + ((uint32_t)(127 - S + 1 - 8) << 23));
  const uint32_t mid = __funnelshift_r(lo, hi, 16);
  float tf[K];
  coeffs<S, K>(lo, mid, hi, rc, tf);
  float init = 0.f;
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const int d = (K - 1 - j) % G;
    init = __fmaf_rn(tf[j], -(float)((1 << (S + d)) + (1 << (S - 1))), init);
  }
  weights_from<S, K, G, 0>(qlo, qhi, rc, tf, init, I);
}

__host__ __device__ inline uint64_t stream_bytes_required(uint64_t bits) {
  return ((bits + 7) / 8 + 15) / 16 * 16 + 16;
}

}  // namespace seedq
