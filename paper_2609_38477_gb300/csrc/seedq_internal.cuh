// Internal definitions of libseedq (sm_103a).  Not part of the C ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/seedq.h"
#include "f32x2.cuh"

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

__host__ __device__ constexpr int rung_S(int code) { return 8 + 2 * (code / 5); }
__host__ __device__ constexpr int rung_K(int code) { return 2 + code % 5; }

// Everything a kernel needs about one layer, passed by value.
struct LayerArgs {
  const uint32_t *stream;   // payload words (little-endian bit string)
  uint64_t stream_words;    // readable 32-bit words of the bound stream buffer
  const uint64_t *row_off;  // R + 1 bit offsets
  const int32_t *brk;       // R x (J-1): first block of row r with rung > j
  const uint64_t *tables;   // nslots x 512 LFSR jump tables
  const int32_t *perm;      // C: block c holds columns perm[8c..8c+7]
  const int32_t *invperm;   // C: position of column j in the permuted order
  const uint16_t *out_vals; // R x n_out binary16
  const int32_t *rowperm;   // R: order in which rows are grouped 32 to a warp
  const uint4 *rowrec;      // R x 2, at row position i (row rowperm[i]): its bit
                            // offset (words 0-1), its breakpoints as int16
                            // pairs (words 2-5, 0x7fff past J - 1) and its bit
                            // count (word 6)
  float *xperm;             // C x n: activations in permuted order, weight-major
  int32_t *counters;        // row groups: arrivals of partial sums (0 between calls)
  float *slots;             // max_ctas x 2 x 32 x 16 partial sums of row groups
  uint32_t *flags;
  int64_t R, C;
  int32_t nb;               // C / 8 blocks per row
  int32_t J;
  int32_t L[kMaxJ];         // block bits per rung
  int32_t dL[kMaxJ - 1];    // L[j + 1] - L[j] for j < J - 1, else 0
  int32_t code[kMaxJ];      // rung_code per rung
  int32_t slot[kMaxJ];      // LFSR table slot per rung
  int32_t nslots;
  int32_t n_out;
  int32_t out_cols[kMaxOutliers];
  uint32_t zero;            // 0; see RungRt
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
  uint4 *d_rowrec;
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

// Entry v of the GF(2) jump table of width S (0 <= v < 512): the first 64
// sequence bits o_0..o_63 from seed v (v < 256) or from seed (v - 256) << 8
// reduced to S bits (zero for S = 8), by the window recurrence
// o_{t+S} = XOR over set bits i of taps of o_{t+i}.  By linearity the prefix
// of any seed s is tab[s & 255] ^ tab[256 + (s >> 8)].
__device__ __forceinline__ uint64_t jump_table_entry(int S, uint32_t taps, int v) {
  const uint32_t seed = (v < 256) ? (uint32_t)v : ((uint32_t)(v - 256) << 8);
  uint64_t q = (uint64_t)(seed & ((1u << S) - 1u));
  if (v >= 256 && S <= 8) q = 0;
  for (int t = S; t < 64; ++t) {
    const uint64_t win = (q >> (t - S)) & (uint64_t)taps;
    const uint64_t bit = (uint64_t)(__popcll(win) & 1);
    q |= bit << t;
  }
  return q;
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

// ---------------------------------------------------------- reconstruction
//
// Eq. codec for one block, exactly: I[i] = sum_j t_j (x_{iK+j} - 2^{S-1}) as an
// fp32 integer and scale = 2^(E-S+1), so w_i = I[i] * scale (exact, |I| < 2^21).
//
// LFSR: the 64-bit sequence prefix Q = o_0..o_63 comes from two GF(2)-linear
// jump tables indexed by the seed's bytes: tab[v] = Q(v), tab[256+v] =
// Q((v mod 2^(S-8)) << 8), so the raw second byte of the field word indexes it
// (for S = 8 the second half is all zero).
//
// Fields: f = bits [S, S+32) of the block puts E at [0, 4) and t_j at
// [4+4j, 8+4j); a 4-bit field read under a fixed exponent gives t_j as a float.
//
// States as floats: Q is shifted left by 23 - S into three words (q2:q1:q0),
// so state x_n sits at bits [23-S, 23) of the 32-bit window starting at bit n
// (a compile-time position); state n-d of the same window lies at
// [23-S-d, 23-d), and masking it and OR-ing exponent 127+S+d gives the float
// 2^(S+d) + x_{n-d}.  A group of G consecutive states of one weight shares one
// window.  An FMA chain from init = -sum_j t_j (2^(S+d_j) + 2^(S-1)) then
// yields I exactly, provided every partial sum stays an integer below 2^24 in
// magnitude; group_size() picks the largest G for which the worst case (all
// |t_j| = 8) satisfies that, and the kernels use the value for S = 16, which
// bounds every smaller width.  S is a run-time value: one code body per K.

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

// Per-rung constants kept in registers, built once per run of blocks.  They
// are derived from a runtime zero so the compiler cannot fold them into
// instruction immediates: a LOP3 takes one immediate at most, and
// (w & mask) | exponent must stay a single LOP3.
template <int K>
struct RungRt {
  static constexpr int G = group_size(16, K);
  static_assert(exact_bound(16, K, G) < (1ll << 24), "FMA chain would round");
  uint32_t S, qs;                 // seed width, 23 - S
  uint32_t e_msk, e_x, sc;        // E field (at bit 0) and the scale's exponent offset
  uint32_t t_msk[K], t_x[K];      // t_j fields
  uint32_t s_msk[G], s_exp[G];    // state windows by offset d within a group
  float cinit[K];                 // -(2^(S+d_j) + 2^(S-1))
  __device__ __forceinline__ RungRt(int S_, uint32_t z) {
    S = (uint32_t)S_;
    qs = (uint32_t)(23 - S_);
    e_msk = 15u ^ z;
    e_x = 8u ^ z;
    sc = ((uint32_t)(120 - S_) << 23) ^ z;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      const int P = (4 + 4 * j <= 19) ? 4 + 4 * j : 4 + 4 * j - 16;
      t_msk[j] = (15u << P) ^ z;
      t_x[j] = ((8u << P) | ((uint32_t)(150 - P) << 23)) ^ z;
      const int d = (K - 1 - j) % G;
      cinit[j] = -(float)((1 << (S_ + d)) + (1 << (S_ - 1)));
    }
#pragma unroll
    for (int d = 0; d < G; ++d) {
      s_msk[d] = ((((1u << S_) - 1u) << (23 - S_)) >> d) ^ z;
      s_exp[d] = ((uint32_t)(127 + S_ + d) << 23) ^ z;
    }
  }
};

// 32 bits of the 96-bit value (q2:q1:q0) starting at bit N (0 <= N < 64).
template <int N>
__device__ __forceinline__ uint32_t qwin3(uint32_t q0, uint32_t q1, uint32_t q2) {
  if constexpr (N == 0) return q0;
  else if constexpr (N < 32) return __funnelshift_r(q0, q1, N);
  else if constexpr (N == 32) return q1;
  else return __funnelshift_r(q1, q2, N - 32);
}

// The chains of weights 2p and 2p + 1 run side by side in the two halves of
// packed f32x2 FMAs (each half rounds as the scalar FMA would, so I is the
// same exact integer).
template <int K, int P, int J>
__device__ __forceinline__ uint64_t state_chain2(uint32_t q0, uint32_t q1, uint32_t q2,
                                                 const RungRt<K> &rc, const uint64_t (&tf2)[K],
                                                 uint64_t acc) {
  if constexpr (J < 0) {
    return acc;
  } else {
    constexpr int G = RungRt<K>::G;
    constexpr int grp = (K - 1 - J) / G;
    constexpr int jt = K - 1 - grp * G;
    constexpr int d = jt - J;
    const uint32_t w0 = qwin3<(2 * P) * K + jt>(q0, q1, q2);
    const uint32_t w1 = qwin3<(2 * P + 1) * K + jt>(q0, q1, q2);
    const uint64_t st = f2_pack(__uint_as_float(lop_and_or(w0, rc.s_msk[d], rc.s_exp[d])),
                                __uint_as_float(lop_and_or(w1, rc.s_msk[d], rc.s_exp[d])));
    acc = f2_fma(tf2[J], st, acc);
    return state_chain2<K, P, J - 1>(q0, q1, q2, rc, tf2, acc);
  }
}

// lo, hi: the block's 64 field bits starting at its first bit.  Ip[p] holds
// (I[2p], I[2p + 1]).
template <int K>
__device__ __forceinline__ void reconstruct_rt2(uint32_t lo, uint32_t hi, const uint64_t *tab,
                                                const RungRt<K> &rc, uint64_t (&Ip)[4], float &scale) {
  // For S = 8 the second table half is all zero, so both lookups are always valid.
  const uint64_t Q = tab[lo & 255u] ^ tab[256 + __byte_perm(lo, 0, 0x4441)];
  const uint32_t qlo = (uint32_t)Q, qhi = (uint32_t)(Q >> 32);
  const uint32_t q0 = qlo << rc.qs;
  const uint32_t q1 = __funnelshift_l(qlo, qhi, rc.qs);
  const uint32_t q2 = __funnelshift_l(qhi, 0u, rc.qs);
  const uint32_t f = __funnelshift_r(lo, hi, rc.S);
  const uint32_t e8 = lop_and_xor(f, rc.e_msk, rc.e_x);
  scale = __uint_as_float(e8 * (1u << 23) + rc.sc);
  float tf[K];
  uint64_t tf2[K];
  uint32_t f2 = 0;
  if constexpr (K > 4) f2 = f >> 16;
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const int P = (4 + 4 * j <= 19) ? 4 + 4 * j : 4 + 4 * j - 16;
    const uint32_t w = (4 + 4 * j <= 19) ? f : f2;
    tf[j] = __uint_as_float(lop_and_xor(w, rc.t_msk[j], rc.t_x[j])) - (float)((1 << (23 - P)) + 8);
    tf2[j] = f2_pack(tf[j], tf[j]);
  }
  float init = 0.f;
#pragma unroll
  for (int j = 0; j < K; ++j) init = __fmaf_rn(tf[j], rc.cinit[j], init);
  const uint64_t init2 = f2_pack(init, init);
  Ip[0] = state_chain2<K, 0, K - 1>(q0, q1, q2, rc, tf2, init2);
  Ip[1] = state_chain2<K, 1, K - 1>(q0, q1, q2, rc, tf2, init2);
  Ip[2] = state_chain2<K, 2, K - 1>(q0, q1, q2, rc, tf2, init2);
  Ip[3] = state_chain2<K, 3, K - 1>(q0, q1, q2, rc, tf2, init2);
}

template <int K>
__device__ __forceinline__ void reconstruct_rt(uint32_t lo, uint32_t hi, const uint64_t *tab,
                                               const RungRt<K> &rc, float (&I)[8], float &scale) {
  uint64_t Ip[4];
  reconstruct_rt2<K>(lo, hi, tab, rc, Ip, scale);
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const float2 v = f2_unpack(Ip[p]);
    I[2 * p] = v.x;
    I[2 * p + 1] = v.y;
  }
}

// ------------------------------------- reconstruction with subnormal states
//
// The same exact integers I[i] of Eq. codec, with fewer logic instructions
// (the fused kernel's form; reconstruct_rt above stays the decoder's).
//
// A 32-bit word whose sign and exponent bits are zero is the float
// m * 2^-149, m its 23-bit mantissa field.  So a state x_n lying at bit
// offset o of a 32-bit window of the sequence (bits [o, o + S), o + S <= 23),
// masked out of the window by a single AND, is the float x_n * 2^(o - 149):
// no exponent has to be inserted and the state need not sit at a fixed
// position.  One window thus serves every state that starts in its first
// 24 - S bits, and Q is used as the tables return it (no shift into exponent
// position):
//   K <= 4: the window at bit 2pK holds the 2K states of weights 2p and 2p+1
//           (offsets j and K + j; 2K + S <= 24 for S <= 16);
//   K >= 5: the window at bit iK holds the K states of weight i (offset j).
//
// The offsets go into the coefficients: tf_j = t_j * 2^(M - j) (M = 108) comes
// straight from the 4-bit field read under a larger exponent, so
// tf_j * x_n 2^(j - 149) = t_j x_n u with u = 2^(M - 149) = 2^-41 for a weight
// at offset j, and 2^K times that for the odd weight of a shared window.
// Every product is exact, every partial sum of a chain is an integer multiple
// of its unit below 2^24 units (|partial| <= 12 K 2^S < 2^23 for S <= 16,
// K <= 6), so each chain yields its I exactly:
//   Ip[p] = (I[2p] u, I[2p+1] u 2^Ko), Ko = K for K <= 4, else 0,
// and scale = 2^(E - S + 1) / u.  The FMAs keep subnormal operands (no .ftz).
// Scaling by powers of two changes no rounding, so a product with x rounds as
// it would on the unscaled I (unless |x| < 2^-85, where u I x is subnormal).
constexpr int kDnM = 108;

__host__ __device__ constexpr int field_pos(int j) { return (4 + 4 * j <= 19) ? 4 + 4 * j : 4 + 4 * j - 16; }
// The float read from field j when t_j = 0 (field value 8 after the XOR):
// 2^(131 - P - j) + 8 * 2^(M - j); any t_j reads as that plus t_j 2^(M - j).
__host__ __device__ constexpr uint32_t dn_tbits(int j) {
  return (8u << field_pos(j)) | ((uint32_t)(150 + kDnM - field_pos(j) - j) << 23);
}
static_assert(150 + kDnM - 4 <= 254, "coefficient exponent out of range");

template <int K>
struct RungDn {
  static constexpr bool kPair = 2 * K + 16 <= 24;
  static constexpr int Ko = kPair ? K : 0;
  uint32_t S;
  uint32_t e_msk, e_x, sc;      // E field (at bit 0) and the scale's exponent offset
  uint32_t t_msk[K], t_x[K];    // t_j fields
  uint32_t m_e[K];              // state masks: offset j
  uint32_t m_o[kPair ? K : 1];  // offset K + j (odd weight of a shared window)
  uint64_t cinit2[K];           // (-2^(S+j-150), -2^(S+j-150+Ko)): the centring -2^(S-1) t_j u
  __device__ __forceinline__ RungDn(int S_, uint32_t z) {
    S = (uint32_t)S_;
    e_msk = 15u ^ z;
    e_x = 8u ^ z;
    sc = ((uint32_t)(120 + 149 - kDnM - S_) << 23) ^ z;
    const uint32_t ms = (1u << S_) - 1u;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      t_msk[j] = (15u << field_pos(j)) ^ z;
      t_x[j] = dn_tbits(j) ^ z;
      m_e[j] = (ms << j) ^ z;
      if constexpr (kPair) m_o[j] = (ms << (K + j)) ^ z;
      // Subnormal: S + j - 1 + Ko <= 22.
      const uint32_t ce = 0x80000000u | (1u << (S_ + j - 1)), co = 0x80000000u | (1u << (S_ + j - 1 + Ko));
      cinit2[j] = ((uint64_t)(co ^ z) << 32) | (uint64_t)(ce ^ z);
    }
  }
  // The same constants as a table entry of 1 + 2K 16-byte words (store), read
  // back by the second constructor.
  static constexpr int kEntry = 1 + 2 * 6;
  __device__ __forceinline__ void store(uint4 *e) const {
    e[0] = make_uint4(S, e_msk, e_x, sc);
#pragma unroll
    for (int j = 0; j < K; ++j) {
      e[1 + 2 * j] = make_uint4(t_msk[j], t_x[j], m_e[j], kPair ? m_o[kPair ? j : 0] : 0u);
      e[2 + 2 * j] = make_uint4((uint32_t)cinit2[j], (uint32_t)(cinit2[j] >> 32), 0u, 0u);
    }
  }
  __device__ __forceinline__ explicit RungDn(const uint4 *e) {
    const uint4 h = e[0];
    S = h.x;
    e_msk = h.y;
    e_x = h.z;
    sc = h.w;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      const uint4 a = e[1 + 2 * j];
      const uint2 b = *reinterpret_cast<const uint2 *>(e + 2 + 2 * j);
      t_msk[j] = a.x;
      t_x[j] = a.y;
      m_e[j] = a.z;
      if constexpr (kPair) m_o[j] = a.w;
      cinit2[j] = ((uint64_t)b.y << 32) | (uint64_t)b.x;
    }
  }
};

// Bits [N, N + 32) of Q = (qhi:qlo), zero past bit 63 (0 <= N < 64).
template <int N>
__device__ __forceinline__ uint32_t qwin2(uint32_t qlo, uint32_t qhi) {
  if constexpr (N == 0) return qlo;
  else if constexpr (N < 32) return __funnelshift_r(qlo, qhi, N);
  else if constexpr (N == 32) return qhi;
  else return qhi >> (N - 32);
}

template <int K, int P, int J>
__device__ __forceinline__ uint64_t dn_chain(uint32_t qlo, uint32_t qhi, const RungDn<K> &rc,
                                             const uint64_t (&tf2)[K], uint64_t acc) {
  if constexpr (J >= K) {
    return acc;
  } else {
    uint32_t se, so;
    if constexpr (RungDn<K>::kPair) {
      const uint32_t w = qwin2<2 * P * K>(qlo, qhi);
      se = w & rc.m_e[J];
      so = w & rc.m_o[J];
    } else {
      se = qwin2<2 * P * K>(qlo, qhi) & rc.m_e[J];
      so = qwin2<(2 * P + 1) * K>(qlo, qhi) & rc.m_e[J];
    }
    acc = f2_fma(tf2[J], f2_pack(__uint_as_float(se), __uint_as_float(so)), acc);
    return dn_chain<K, P, J + 1>(qlo, qhi, rc, tf2, acc);
  }
}

// lo, hi: the block's 64 field bits starting at its first bit.
template <int K>
__device__ __forceinline__ void reconstruct_dn(uint32_t lo, uint32_t hi, const uint64_t *tab,
                                               const RungDn<K> &rc, uint64_t (&Ip)[4], float &scale) {
  // For S = 8 the second table half is all zero, so both lookups are always valid.
  const uint64_t Q = tab[lo & 255u] ^ tab[256 + __byte_perm(lo, 0, 0x4441)];
  const uint32_t qlo = (uint32_t)Q, qhi = (uint32_t)(Q >> 32);
  const uint32_t f = __funnelshift_r(lo, hi, rc.S);
  const uint32_t e8 = lop_and_xor(f, rc.e_msk, rc.e_x);
  scale = __uint_as_float(e8 * (1u << 23) + rc.sc);
  uint64_t tf2[K];
  uint32_t f2 = 0;
  if constexpr (K > 4) f2 = f >> 16;
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const uint32_t w = (4 + 4 * j <= 19) ? f : f2;
    const float tf = __uint_as_float(lop_and_xor(w, rc.t_msk[j], rc.t_x[j])) - __uint_as_float(dn_tbits(j));
    tf2[j] = f2_pack(tf, tf);
  }
  uint64_t init2 = f2_mul(tf2[0], rc.cinit2[0]);
#pragma unroll
  for (int j = 1; j < K; ++j) init2 = f2_fma(tf2[j], rc.cinit2[j], init2);
  Ip[0] = dn_chain<K, 0, 0>(qlo, qhi, rc, tf2, init2);
  Ip[1] = dn_chain<K, 1, 0>(qlo, qhi, rc, tf2, init2);
  Ip[2] = dn_chain<K, 2, 0>(qlo, qhi, rc, tf2, init2);
  Ip[3] = dn_chain<K, 3, 0>(qlo, qhi, rc, tf2, init2);
}


// ------------------------------------------------- fp64 division, integer pipes
//
// a / b rounded to nearest (IEEE), for b normal and a normal or zero with a
// normal quotient, computed with 64-bit integer instructions only.  With the
// significands ma, mb in [2^52, 2^53), the quotient's significand is
// q = floor(ma * 2^s / mb) for s = 52 (ma >= mb) or 53, rounded up when twice
// the remainder exceeds mb (binary division never lands exactly halfway).  q
// comes from an estimate of 2^116 / mb (an fp32 reciprocal refined by two
// Newton steps in fixed point) and is then corrected against the exact
// 128-bit remainder, so the estimate only has to be within a few units.  The
// method is Newton-Raphson refinement of a reciprocal approximation followed
// by quotient correction from the exact remainder, as in the literature on
// division with a precomputed reciprocal (Granlund and Montgomery, "Division
// by invariant integers using multiplication", PLDI 1994; Markstein, "IA-64
// and Elementary Functions", 2000).  A GPU test compares it bit for bit with
// the hardware division on random and edge operands.
struct DivRecip {
  double b;      // the divisor (for the rare operands handled by hardware division)
  uint64_t d;    // significand of b
  uint64_t inv;  // ~ 2^116 / d
  int e;         // unbiased exponent of b
  uint64_t sign; // sign bit of b
};

__device__ __forceinline__ void mul128(uint64_t a, uint64_t b, uint64_t &hi, uint64_t &lo) {
  hi = __umul64hi(a, b);
  lo = a * b;
}

__device__ __forceinline__ DivRecip div_recip(double b) {
  const uint64_t bb = (uint64_t)__double_as_longlong(b);
  DivRecip r;
  r.b = b;
  r.sign = bb >> 63;
  r.e = (int)((bb >> 52) & 2047) - 1023;
  r.d = (bb & ((1ull << 52) - 1)) | (1ull << 52);
  // fp32 estimate of 1/d from d's top 24 bits: d ~ (d >> 29) * 2^29.
  const float df = __uint_as_float((uint32_t)((r.d >> 29) & 0x7fffffu) | ((uint32_t)(127 + 52) << 23));
  const uint32_t rb = __float_as_uint(__frcp_rn(df));
  const int er = (int)(rb >> 23) - 127;             // -53 or -52
  const uint64_t m = (rb & 0x7fffffu) | 0x800000u;  // 1/d ~ m * 2^(er - 23)
  const int sh = 116 + er - 23;                      // inv ~ m * 2^sh, sh in {40, 41}
  uint64_t inv = sh >= 41 ? ~0ull : (m << sh);
  // Two Newton steps: inv += inv * (2^116 - d * inv) / 2^116.
#pragma unroll
  for (int it = 0; it < 2; ++it) {
    uint64_t phi, plo;
    mul128(r.d, inv, phi, plo);  // d * inv, around 2^116
    const uint64_t two116 = 1ull << 52;  // 2^116 as (hi = 2^52, lo = 0)
    bool neg;
    uint64_t ehi, elo;
    if (phi >= two116) {
      neg = true;
      elo = plo;
      ehi = phi - two116;  // d*inv - 2^116
    } else {
      neg = false;
      elo = 0ull - plo;
      ehi = two116 - phi - (plo != 0 ? 1ull : 0ull);
    }
    // correction = inv * e / 2^116, with e >> 52 (e < 2^116).
    const uint64_t e52 = (ehi << 12) | (elo >> 52);
    const uint64_t corr = __umul64hi(inv, e52);
    inv = neg ? inv - corr : inv + corr;
  }
  r.inv = inv;
  return r;
}

__device__ __forceinline__ double div_rn(double a, const DivRecip &R) {
  const uint64_t ab = (uint64_t)__double_as_longlong(a);
  const uint64_t sign = (ab >> 63) ^ R.sign;
  if ((ab & 0x7fffffffffffffffull) == 0) return __longlong_as_double((long long)(sign << 63));
  const int ea = (int)((ab >> 52) & 2047) - 1023;
  const uint64_t ma = (ab & ((1ull << 52) - 1)) | (1ull << 52);
  const int s = ma >= R.d ? 52 : 53;
  int e = ea - R.e - (s - 52);
  // Subnormal or non-finite operands, or a quotient near the end of the
  // exponent range: hardware division (never taken by the encoder's values).
  if (ea == -1023 || ea == 1024 || R.e == -1023 || R.e == 1024 || e < -1021 || e > 1022) return a / R.b;
  // N = ma * 2^s as 128 bits.
  const uint64_t nhi = ma >> (64 - s), nlo = ma << s;
  const uint64_t n42 = (nhi << 22) | (nlo >> 42);
  uint64_t q = __umul64hi(n42, R.inv) >> 10;
  // Exact remainder N - q * d, then correct q by whole units.
  uint64_t phi, plo;
  mul128(q, R.d, phi, plo);
  long long rhi = (long long)(nhi - phi - (nlo < plo ? 1ull : 0ull));
  uint64_t rlo = nlo - plo;
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    if (rhi < 0) {  // remainder negative: q too large
      --q;
      const uint64_t t = rlo + R.d;
      rhi += (t < rlo) ? 1 : 0;
      rlo = t;
    }
  }
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    if (rhi > 0 || rlo >= R.d) {  // remainder >= d: q too small
      ++q;
      rhi -= (rlo < R.d) ? 1 : 0;
      rlo -= R.d;
    }
  }
  if (2 * rlo > R.d) ++q;  // round to nearest (no ties)
  if (q == (1ull << 53)) {
    q = 1ull << 52;
    ++e;
  }
  return __longlong_as_double((long long)((sign << 63) | ((uint64_t)(e + 1023) << 52) | (q - (1ull << 52))));
}

__host__ __device__ inline uint64_t stream_bytes_required(uint64_t bits) {
  return ((bits + 7) / 8 + 15) / 16 * 16 + 16;
}

}  // namespace seedq
