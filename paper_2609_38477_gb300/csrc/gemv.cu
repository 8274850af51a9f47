// Fused reconstruction x matrix-vector product: y = W_hat x, and the decode-batch
// skinny GEMM Y = X W_hat^T (n <= 16), for one tensor or for several tensors
// in one launch (the tensors of a decode step are independent: Alg. 2 decodes
// each tensor on its own, in no fixed order).  W_hat is never written to memory; HBM carries only
// the compressed streams, the plan rows and x / y.
//
// Layout: a lane owns a row.  A warp takes 32 rows (a row group, in the plan's
// row order, which puts rows with equal or nearby rung breakpoints together)
// and walks their blocks column by column, so all lanes usually sit at the
// same rung: control flow is uniform and the activations of a column are one
// broadcast read.  A warp stages the stream bytes of its 32 rows, a few
// columns at a time, into shared memory with cp.async (double-buffered),
// together with the column slice of the activations (permuted once per call
// into scratch by a small pre-kernel).
//
// Work split: all (tensor, row group, block) units in one sequence, cut into
// one contiguous range per CTA (one CTA per SM) of equal modeled cost.  A CTA
// processes its range in rounds of a few row groups of one tensor; the round's
// stages are dealt round-robin to its 12 warps, whose partial sums are added
// in warp order in shared memory.  A row group cut by a CTA boundary leaves
// one partial sum per CTA in scratch; the CTA that arrives last adds them in
// CTA order.  No result depends on timing.
#include <cuda_fp16.h>
#include <string.h>

#include <cstddef>
#include <new>
#include <vector>

#include "cp_async.cuh"
#include "device_once.h"
#include "f32x2.cuh"
#include "seedq_internal.cuh"

namespace seedq {

constexpr int kWarps = 12;
constexpr int kThreads = kWarps * 32;
constexpr int kMaxTensors = 8;
constexpr int kMaxCtas = 256;

template <int NB>
struct Cfg {
  // Columns per stage and row groups per round: the widest stage for which
  // 12 warps' double buffers, the jump tables and the round's partial sums
  // fit in shared memory (wider stages amortize staging and bookkeeping).
  static constexpr int ST = NB == 1 ? 27 : NB == 2 ? 21 : NB == 4 ? 15 : NB == 8 ? 12 : 7;
  static constexpr int RG = NB == 1 ? 8 : NB <= 4 ? 4 : 1;
  // 16-byte pieces per staged row: ST blocks of at most 44 bits, the 96-bit
  // read-ahead of the last block, and up to 15 + 15 bytes of alignment.
  static constexpr int PIECES = (ST * 44 / 8 + 12 + 30 + 15) / 16 + 1;
  // Row stride in words: 16-byte aligned with an odd number of 16-byte pieces,
  // so 8 consecutive rows start in 8 different bank groups.
  static constexpr int RW = (PIECES % 2) ? PIECES * 4 : PIECES * 4 + 4;
  static constexpr int STREAM_WORDS = 2 * 32 * RW;  // per warp, double-buffered
  static constexpr int XFLOATS = 2 * ST * 8 * NB;   // per warp, double-buffered
  static constexpr int WARP_BYTES = STREAM_WORDS * 4 + XFLOATS * 4;
};

struct TensorArgs {
  LayerArgs p;
  const uint16_t *x;      // n x C bf16, original column order
  float *y;               // n x R
  int64_t ubegin;         // first unit of this tensor in the launch's sequence
  uint64_t stream_bytes;  // readable bytes of the bound stream buffer
  int64_t cpre, rpre;     // layer sets: columns and rows of the tensors before it
};

// One launch over several tensors.  The descriptors and the CTA ranges are
// either inline (seedq_gemm_multi, up to kMaxTensors) or, for a layer set,
// in device memory, with every tensor's x and y at fixed offsets of one
// activation and one output buffer.
struct MultiArgs {
  TensorArgs t[kMaxTensors];
  int nt;
  int n;
  int ctas;
  uint32_t zero;  // 0 at run time; keeps per-rung constants out of immediates
  int64_t cta_begin[kMaxCtas + 1];
  const TensorArgs *tens;  // layer set: nt descriptors (else t)
  const int64_t *cbd;      // layer set: ctas + 1 range starts (else cta_begin)
  const uint16_t *Xall;    // layer set: x of tensor i at Xall + n * cpre_i
  float *Yall;             // layer set: y of tensor i at Yall + n * rpre_i
};

__host__ __device__ inline int batch_template(int n) {
  return n <= 1 ? 1 : n <= 2 ? 2 : n <= 4 ? 4 : n <= 8 ? 8 : 16;
}

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }

// CTA whose range holds unit u (cb: the ctas + 1 range starts).
__device__ __forceinline__ int cta_of(const int64_t *cb, int ctas, int64_t u) {
  int lo = 0, hi = ctas - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (cb[mid] <= u) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// One block: reconstruct its 8 weights and add scale * sum_i I_i x_b[i] to
// acc[b].  xc holds the block's activations weight-major, NB per weight
// (xc[i * NB + b]).  The reconstruction leaves (I[2p], I[2p+1]) in the two
// halves of a packed pair, the odd half 2^Ko times larger (reconstruct_dn).
// At NB = 1 the products run in those halves, which are added with the odd
// one scaled back; at NB >= 2 two batch columns share each packed
// instruction, in one chain over the even and one over the odd weights.
template <int K, int NB>
__device__ __forceinline__ void block_fma(const uint32_t (&w)[3], uint32_t sh, const uint64_t *tab,
                                          const RungDn<K> &rc, const float *xc, float (&acc)[NB]) {
  const uint32_t lo = __funnelshift_r(w[0], w[1], sh);  // the shift is taken mod 32
  const uint32_t hi = __funnelshift_r(w[1], w[2], sh);
  uint64_t I2[4];
  float scale;
  reconstruct_dn<K>(lo, hi, tab, rc, I2, scale);
  constexpr float kOdd = 1.0f / (float)(1 << RungDn<K>::Ko);
  if constexpr (NB == 1) {
    const ulonglong2 xa = *reinterpret_cast<const ulonglong2 *>(xc);
    const ulonglong2 xb = *reinterpret_cast<const ulonglong2 *>(xc + 4);
    uint64_t s2 = f2_mul(I2[0], xa.x);
    s2 = f2_fma(I2[1], xa.y, s2);
    s2 = f2_fma(I2[2], xb.x, s2);
    s2 = f2_fma(I2[3], xb.y, s2);
    const float2 sv = f2_unpack(s2);
    acc[0] = __fmaf_rn(scale, __fmaf_rn(sv.y, kOdd, sv.x), acc[0]);
  } else {
    const uint64_t *x2 = reinterpret_cast<const uint64_t *>(xc);  // pairs of batch columns
    uint64_t Ip[8];
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const float2 v = f2_unpack(I2[p]);
      Ip[2 * p] = f2_pack(v.x, v.x);
      Ip[2 * p + 1] = f2_pack(v.y, v.y);
    }
    const uint64_t sp = f2_pack(scale, scale), ko = f2_pack(kOdd, kOdd);
#pragma unroll
    for (int q = 0; q < NB / 2; ++q) {
      uint64_t s0 = f2_mul(Ip[0], x2[0 * (NB / 2) + q]), s1 = f2_mul(Ip[1], x2[1 * (NB / 2) + q]);
      s0 = f2_fma(Ip[2], x2[2 * (NB / 2) + q], s0);
      s1 = f2_fma(Ip[3], x2[3 * (NB / 2) + q], s1);
      s0 = f2_fma(Ip[4], x2[4 * (NB / 2) + q], s0);
      s1 = f2_fma(Ip[5], x2[5 * (NB / 2) + q], s1);
      s0 = f2_fma(Ip[6], x2[6 * (NB / 2) + q], s0);
      s1 = f2_fma(Ip[7], x2[7 * (NB / 2) + q], s1);
      const uint64_t a = f2_fma(sp, f2_fma(s1, ko, s0), f2_pack(acc[2 * q], acc[2 * q + 1]));
      acc[2 * q] = __uint_as_float((uint32_t)a);
      acc[2 * q + 1] = __uint_as_float((uint32_t)(a >> 32));
    }
  }
}

template <int K, int NB>
__device__ __forceinline__ void run_cols(const uint4 *rent, const uint32_t *rowbuf, uint32_t &pos, int n,
                                         const uint64_t *tab, const float *xc, float (&acc)[NB]) {
  const RungDn<K> rc(rent);
  const uint32_t L = rc.S + (uint32_t)(4 * K + 4);
  uint32_t w[3];
  {
    const uint32_t *q = rowbuf + (pos >> 5);
    w[0] = q[0];
    w[1] = q[1];
    w[2] = q[2];
  }
  for (int i = 0; i < n; ++i) {
    const uint32_t cur[3] = {w[0], w[1], w[2]};
    const uint32_t sh = pos;
    pos += L;
    {
      // Also after the last block: the words past a stage's end stay inside
      // the lane's RW-word row buffer (at most (127 + ST * 44) / 32 + 3 words),
      // and what they hold is not used.
      const uint32_t *q = rowbuf + (pos >> 5);
      w[0] = q[0];
      w[1] = q[1];
      w[2] = q[2];
    }
    block_fma<K, NB>(cur, sh, tab, rc, xc + i * 8 * NB, acc);
  }
}

template <int NB>
__device__ __forceinline__ void dispatch_cols(int code, const uint4 *rent, const uint32_t *rowbuf,
                                              uint32_t &pos, int n, const uint64_t *tab, const float *xc,
                                              float (&acc)[NB]) {
  switch (rung_K(code)) {
    case 2: run_cols<2, NB>(rent, rowbuf, pos, n, tab, xc, acc); break;
    case 3: run_cols<3, NB>(rent, rowbuf, pos, n, tab, xc, acc); break;
    case 4: run_cols<4, NB>(rent, rowbuf, pos, n, tab, xc, acc); break;
    case 5: run_cols<5, NB>(rent, rowbuf, pos, n, tab, xc, acc); break;
    default: run_cols<6, NB>(rent, rowbuf, pos, n, tab, xc, acc); break;
  }
}

// The per-rung constants of RungDn for every rung of a tensor (thread j < J
// writes rung j's entry).
__device__ __forceinline__ void store_rung_entries(const LayerArgs &p, uint32_t z, uint4 *rdn) {
  const int j = threadIdx.x;
  if (j >= p.J) return;
  const int code = p.code[j], S = rung_S(code);
  uint4 *e = rdn + j * RungDn<2>::kEntry;
  switch (rung_K(code)) {
    case 2: RungDn<2>(S, z).store(e); break;
    case 3: RungDn<3>(S, z).store(e); break;
    case 4: RungDn<4>(S, z).store(e); break;
    case 5: RungDn<5>(S, z).store(e); break;
    default: RungDn<6>(S, z).store(e); break;
  }
}

// Bits of the lane's row before blocks cs and ce.  Rung j spans blocks
// [bk[j-1], bk[j]) and the breakpoints rise along the row, so the bits before
// block x are L[0] x plus, for every breakpoint below x, the rate step dL[j]
// times the blocks past it.  bw: the row's breakpoints as int16 pairs (0x7fff,
// above every block index, past J - 1, where dL is zero).
__device__ __forceinline__ void lane_bits_before(const uint32_t (&bw)[4], const LayerArgs &p, int cs,
                                                 int ce, uint32_t &s_cs, uint32_t &s_ce) {
  s_cs = (uint32_t)p.L[0] * (uint32_t)cs;
  s_ce = (uint32_t)p.L[0] * (uint32_t)ce;
#pragma unroll
  for (int j = 0; j < kMaxJ - 1; ++j) {
    const int b = (int)((bw[j >> 1] >> (16 * (j & 1))) & 0xffffu);
    s_cs += (uint32_t)p.dL[j] * (uint32_t)max(cs - b, 0);
    s_ce += (uint32_t)p.dL[j] * (uint32_t)max(ce - b, 0);
  }
}

// A piece of a round: blocks [ca, cb) of row group g of the round's tensor.
struct Piece {
  int64_t g;
  int ca, cb;
};

// The stages of a round (pieces cut into ST-column stages, in order) dealt
// round-robin to the CTA's warps; lane = row of the stage's row group.  Each
// buffer slot carries the row data of the stage staged into it.  A warp's sums
// go to comb[piece][warp][lane] whenever its next stage is in another piece.
template <int NB>
__device__ __forceinline__ void warp_round(const TensorArgs &T, int n, const uint4 *rdn,
                                           const uint64_t *tabs, uint32_t *sbuf, float *xbuf,
                                           const uint4 *rrec, const Piece *pcs, const int *pst, int np,
                                           int nst_total,
                                           float *comb, int warp, int lane) {
  using CF = Cfg<NB>;
  const LayerArgs &p = T.p;
  const int J = p.J, nb = p.nb;
  if (warp >= nst_total) return;
  const uint8_t *gstream = reinterpret_cast<const uint8_t *>(p.stream);
  int piece_of[2] = {0, 0}, cs_of[2] = {0, 0}, ce_of[2] = {0, 0};
  int jr_of[2] = {0, 0}, nxt_of[2] = {0, 0};
  uint32_t pos0[2] = {0, 0};

  int pi_cur = 0;  // piece of the last stage issued (a warp's stages rise)
  auto issue = [&](int t, int sb) {
    while (pi_cur + 1 < np && t >= pst[pi_cur + 1]) ++pi_cur;
    const int pi = pi_cur;
    const int cs = pcs[pi].ca + (t - pst[pi]) * CF::ST, ce = min(pcs[pi].cb, cs + CF::ST);
    // The lane's row record (bit offset, breakpoints), staged for the round.
    const uint4 m0 = rrec[(pi * 32 + lane) * 2], m1 = rrec[(pi * 32 + lane) * 2 + 1];
    const uint64_t roff = (uint64_t)m0.x | ((uint64_t)m0.y << 32);
    const uint32_t bw[4] = {m0.z, m0.w, m1.x, m1.y};
    uint32_t s_cs, s_ce;
    lane_bits_before(bw, p, cs, ce, s_cs, s_ce);
    // A row's last stage ends where its record says the row ends.
    if (ce == nb && s_ce != m1.z) atomicOr(p.flags, 1u);
    // Rung of block cs (breakpoints at or below it) and the next breakpoint.
    int jr0 = 0, nx0 = nb;
#pragma unroll
    for (int j = 0; j < kMaxJ - 1; ++j) {
      const int b = (int)((bw[j >> 1] >> (16 * (j & 1))) & 0xffffu);  // 0x7fff past J - 1
      jr0 += (b <= cs) ? 1 : 0;
      if (b > cs) nx0 = min(nx0, b);
    }
    const uint64_t bit_cs = roff + s_cs;
    const uint64_t b_lo = (bit_cs >> 3) & ~(uint64_t)15;
    uint64_t b_hi = (roff + s_ce + 96 + 7) >> 3;
    b_hi = (b_hi + 15) & ~(uint64_t)15;
    if (b_hi > T.stream_bytes) {
      // A stage reaching past the readable stream: the plan disagrees with
      // the bound buffer.  Read only what is there and report it.
      atomicOr(p.flags, 1u);
      b_hi = T.stream_bytes & ~(uint64_t)15;
    }
    const int npc = b_hi > b_lo ? (int)min((uint64_t)CF::PIECES, (b_hi - b_lo) >> 4) : 0;
    const uint32_t p0 = (uint32_t)(bit_cs - b_lo * 8);
    if (sb) {
      piece_of[1] = pi; cs_of[1] = cs; ce_of[1] = ce; pos0[1] = p0; jr_of[1] = jr0; nxt_of[1] = nx0;
    } else {
      piece_of[0] = pi; cs_of[0] = cs; ce_of[0] = ce; pos0[0] = p0; jr_of[0] = jr0; nxt_of[0] = nx0;
    }
    uint32_t *rows = sbuf + sb * 32 * CF::RW;
#pragma unroll
    for (int pc = 0; pc < CF::PIECES; ++pc)
      if (pc < npc) cp_async16(rows + lane * CF::RW + pc * 4, gstream + b_lo + 16 * pc);
    float *xs = xbuf + sb * CF::ST * 8 * NB;
    // Activations of the stage's columns: contiguous in the weight-major
    // scratch layout (NB values per weight).
    const int nq = (ce - cs) * 2 * NB;  // 16-byte pieces
    for (int q = lane; q < nq; q += 32)
      cp_async16(xs + q * 4, p.xperm + (int64_t)cs * 8 * NB + q * 4);
    cp_async_commit();
  };

  float acc[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) acc[b] = 0.f;
  int acc_piece = -1;
  issue(warp, 0);
  int it = 0;
  for (int t = warp; t < nst_total; t += kWarps, ++it) {
    const int sb = it & 1;
    if (t + kWarps < nst_total) {
      issue(t + kWarps, sb ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncwarp();
    const int pi = sb ? piece_of[1] : piece_of[0];
    const int cs = sb ? cs_of[1] : cs_of[0], ce = sb ? ce_of[1] : ce_of[0];
    uint32_t pos = sb ? pos0[1] : pos0[0];
    if (pi != acc_piece) {
      if (acc_piece >= 0) {
#pragma unroll
        for (int b = 0; b < NB; ++b) comb[((acc_piece * kWarps + warp) * 32 + lane) * NB + b] += acc[b];
      }
#pragma unroll
      for (int b = 0; b < NB; ++b) acc[b] = 0.f;
      acc_piece = pi;
    }
    // The lane's breakpoints (int16, after the 8-byte bit offset of its record).
    const int16_t *mybk = reinterpret_cast<const int16_t *>(rrec + (pi * 32 + lane) * 2) + 4;
    const uint32_t *rowbuf = sbuf + sb * 32 * CF::RW + lane * CF::RW;
    const float *xs = xbuf + sb * CF::ST * 8 * NB;
    int jr = sb ? jr_of[1] : jr_of[0];
    int nxt = sb ? nxt_of[1] : nxt_of[0];
    // Passes over the stage's columns, each one run of blocks per lane at one
    // rung, all through a single call site (one inlined copy of the rung
    // loops keeps the instruction working set small).  Where all rows sit at
    // one rung a pass is a run of columns shared by the 32 lanes; from the
    // first column where they differ to the end of the stage there is one
    // pass per rung present, each lane running over its own columns at that
    // rung (rungs rise along a row, so a lane's blocks stay in stream order).
    int c = cs;
    int rr = -1, jhi = 0;
    while (true) {
      int j, cnt, xo;
      if (rr < 0) {
        if (c >= ce) break;
        const int jmin = __reduce_min_sync(0xffffffffu, jr), jmax = __reduce_max_sync(0xffffffffu, jr);
        if (jmin == jmax) {
          const int run_end = min((int)__reduce_min_sync(0xffffffffu, (unsigned)nxt), ce);
          j = jmin;
          cnt = run_end - c;
          xo = c - cs;
          c = run_end;
          while (jr < J - 1 && nxt <= c) {
            ++jr;
            nxt = (jr < J - 1) ? mybk[jr] : nb;
          }
        } else {
          jhi = jr;
          while (jhi < J - 1 && mybk[jhi] <= ce - 1) ++jhi;
          jhi = __reduce_max_sync(0xffffffffu, jhi);
          rr = jmin;
          continue;
        }
      } else {
        if (rr > jhi) break;
        const int ra = max(c, rr > 0 ? mybk[rr - 1] : 0);
        const int rb = min(ce, rr < J - 1 ? mybk[rr] : nb);
        j = rr++;
        cnt = rb > ra ? rb - ra : 0;
        xo = cnt > 0 ? ra - cs : 0;
        if (!__any_sync(0xffffffffu, cnt > 0)) continue;
      }
      dispatch_cols<NB>(p.code[j], rdn + j * RungDn<2>::kEntry, rowbuf, pos, cnt,
                        tabs + p.slot[j] * 512, xs + xo * 8 * NB, acc);
    }
    __syncwarp();
  }
  if (acc_piece >= 0) {
#pragma unroll
    for (int b = 0; b < NB; ++b) comb[((acc_piece * kWarps + warp) * 32 + lane) * NB + b] += acc[b];
  }
}

// Outlier epilogue: y_b[r] += sum_o W16[r, col_o] x_b[col_o] (Sec. 3.5).
__device__ __forceinline__ float outlier_term(const LayerArgs &p, const uint16_t *x, int64_t r, int b) {
  float s = 0.f;
  for (int o = 0; o < p.n_out; ++o) {
    const float w = __half2float(__ushort_as_half(p.out_vals[r * p.n_out + o]));
    s = __fmaf_rn(w, bf16_to_f32(x[(int64_t)b * p.C + p.out_cols[o]]), s);
  }
  return s;
}

// kSet: descriptors in device memory (a layer set), copied per round into
// shared memory; otherwise read straight from the parameter block, whose
// fields the instructions take as constant-bank operands (measurably faster
// for the per-stage bookkeeping at small stages).
template <int NB, bool kSet>
__global__ void __launch_bounds__(kThreads, 1) k_gemv(const __grid_constant__ MultiArgs a) {
  using CF = Cfg<NB>;
  extern __shared__ __align__(16) uint64_t smem[];
  uint64_t *tabs = smem;
  uint8_t *wbase = reinterpret_cast<uint8_t *>(smem + kTableSlots * 512);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint8_t *mine = wbase + warp * CF::WARP_BYTES;
  uint32_t *sbuf = reinterpret_cast<uint32_t *>(mine);
  float *xbuf = reinterpret_cast<float *>(mine + CF::STREAM_WORDS * 4);
  float *comb = reinterpret_cast<float *>(wbase + kWarps * CF::WARP_BYTES);  // RG x kWarps x 32 x NB
  uint4 *rrec = reinterpret_cast<uint4 *>(comb + CF::RG * kWarps * 32 * NB);  // RG x 32 x 2 row records
  {
    // The jump tables depend only on S, so any tensor's copy serves all.
    const uint4 *src = reinterpret_cast<const uint4 *>((kSet ? a.tens : a.t)[0].p.tables);
    uint4 *dst = reinterpret_cast<uint4 *>(tabs);
    for (int i = threadIdx.x; i < kTableSlots * 256; i += kThreads) dst[i] = __ldg(src + i);
  }
  // The permuted activations come from the pre-kernel launched just before.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int cta = blockIdx.x;
  const TensorArgs *tens = kSet ? a.tens : a.t;
  const int64_t *cb = kSet ? a.cbd : a.cta_begin;
  const int64_t u0 = cb[cta], u1 = cb[cta + 1];
  int64_t u = u0;
  bool first = true;
  // The round's tensor descriptor, copied to shared memory (for a layer set
  // with its x and y pointers filled in).
  __shared__ TensorArgs sT;
  constexpr int kTWords = sizeof(TensorArgs) / 4;
  static_assert(sizeof(TensorArgs) % 8 == 0, "descriptor size");
  constexpr int kXWord = offsetof(TensorArgs, x) / 4, kYWord = offsetof(TensorArgs, y) / 4;
  // Row groups cut by this CTA's range (at most two: where the range starts
  // and where it ends inside a group): their partial sums go to slots during
  // the rounds and are finished after the last round.  A: slot 0, B: slot 1.
  int cutA_ti = -1, cutB_ti = -1, warpB = 0;
  int64_t cutA_g = 0, cutB_g = 0;
  int32_t crowA = -1, crowB = -1;
  int ti = 0;
  {
    int lo = 0, hi = a.nt - 1;  // last tensor whose first unit is <= u0
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (tens[mid].ubegin <= u0) lo = mid;
      else hi = mid - 1;
    }
    ti = lo;
  }
  while (u < u1) {
    while (ti + 1 < a.nt && tens[ti + 1].ubegin <= u) ++ti;
    if constexpr (kSet) {
      const uint32_t *srcw = reinterpret_cast<const uint32_t *>(tens + ti);
      uint32_t *dstw = reinterpret_cast<uint32_t *>(&sT);
      const uint64_t xv = (uint64_t)(a.Xall + (int64_t)a.n * tens[ti].cpre);
      const uint64_t yv = (uint64_t)(a.Yall + (int64_t)a.n * tens[ti].rpre);
      for (int w = threadIdx.x; w < kTWords; w += kThreads) {
        uint32_t v = srcw[w];
        if (w == kXWord) v = (uint32_t)xv;
        if (w == kXWord + 1) v = (uint32_t)(xv >> 32);
        if (w == kYWord) v = (uint32_t)yv;
        if (w == kYWord + 1) v = (uint32_t)(yv >> 32);
        dstw[w] = v;
      }
    }
    const TensorArgs &T = kSet ? sT : a.t[ti];
    const LayerArgs &p = T.p;
    const int64_t tub = tens[ti].ubegin;
    const int tnb = tens[ti].p.nb;
    const int64_t tend = (ti + 1 < a.nt) ? tens[ti + 1].ubegin : cb[a.ctas];
    const int64_t rend = min(u1, tend);
    // The next round: up to RG row groups of this tensor.
    // (In shared memory: the stage issue indexes it by a runtime piece number.)
    __shared__ Piece pcs[8];
    __shared__ int pst[8];  // first stage of each piece in the round's stage order
    static_assert(CF::RG <= 8, "round size");
    int np = 0, nst_total = 0;
    int64_t uu = u;
    const int ck = threadIdx.x >> 5, cln = threadIdx.x & 31;
    int64_t cg = 0;
    // Pieces whose row records this thread stages (record words i, i + kThreads).
    const int rk0 = threadIdx.x >> 6, rk1 = (threadIdx.x + kThreads) >> 6;
    int64_t rg0 = 0, rg1 = 0;
    bool any_cut = false;  // the same in every thread
    while (uu < rend && np < CF::RG) {
      const int64_t lu = uu - tub;
      const int64_t g = lu / tnb;
      const int ca = (int)(lu - g * tnb);
      const int cbk = (int)min((int64_t)tnb, ca + (rend - uu));
      if (threadIdx.x == 0) {
        pcs[np] = Piece{g, ca, cbk};
        pst[np] = nst_total;
      }
      if (np == ck) cg = g;
      if (np == rk0) rg0 = g;
      if (np == rk1) rg1 = g;
      any_cut |= !(ca == 0 && cbk == tnb);
      nst_total += (cbk - ca + CF::ST - 1) / CF::ST;
      ++np;
      uu += cbk - ca;
    }
    // The output rows of the round, loaded now (thread t < 32 np: row t % 32
    // of piece t / 32): the loads complete during the round; volatile keeps
    // them ahead of the round's copies.
    // (From the descriptor in the parameter block or device memory: for a layer
    // set the shared copy sT is still being written by other threads here.)
    __shared__ int32_t srow[8 * 32];
    int32_t crow = -1;
    const int32_t *trowperm = tens[ti].p.rowperm;
    if (ck < np && cg * 32 + cln < tens[ti].p.R) {
      const int32_t *ap = trowperm + cg * 32 + cln;
      asm volatile("{\n\t.reg .u64 ga;\n\tcvta.to.global.u64 ga, %1;\n\tld.global.nc.b32 %0, [ga];\n\t}"
                   : "=r"(crow) : "l"(ap));
    }
    for (int i = threadIdx.x; i < np * kWarps * 32 * NB; i += kThreads) comb[i] = 0.f;
    __shared__ uint4 rdn[kMaxJ * RungDn<2>::kEntry];
    store_rung_entries(tens[ti].p, a.zero, rdn);
    // The round's row records (32 bytes per row of each piece; rows past R
    // repeat the group's first row), read once per round.
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = threadIdx.x + h * kThreads;
      const int k = h ? rk1 : rk0;
      if (k < np) {
        const int64_t r0 = (h ? rg1 : rg0) * 32, ridx = r0 + ((i >> 1) & 31);
        rrec[i] = __ldg(tens[ti].p.rowrec + 2 * (ridx < tens[ti].p.R ? ridx : r0) + (i & 1));
      }
    }
    __syncthreads();
    warp_round<NB>(T, a.n, rdn, tabs, sbuf, xbuf, rrec, pcs, pst, np, nst_total, comb, warp, lane);
    if (ck < np) srow[threadIdx.x] = crow;
    __syncthreads();
    // Row sums of the round's pieces (warps added in warp order), every (piece,
    // row, batch column) at once: full row groups go to y, cut ones to this
    // CTA's partial-sum slot (slot 0: the first piece of the CTA's range,
    // slot 1: its last piece).
    for (int i = threadIdx.x; i < np * 32 * NB; i += kThreads) {
      const int k = i / (32 * NB), rem = i - k * 32 * NB, b = rem % NB;
      float v = 0.f;
      for (int w = 0; w < kWarps; ++w) v += comb[(k * kWarps + w) * 32 * NB + rem];
      if (pcs[k].ca == 0 && pcs[k].cb == p.nb) {
        const int32_t rr = srow[k * 32 + rem / NB];
        if (rr >= 0 && b < a.n) T.y[(int64_t)b * p.R + rr] = v + outlier_term(p, T.x, rr, b);
      } else {
        const int sidx = (k == 0 && first) ? 0 : 1;
        p.slots[((int64_t)cta * 2 + sidx) * 32 * kMaxBatch + rem] = v;
      }
    }
    if (any_cut) {
      const bool c0 = first && !(pcs[0].ca == 0 && pcs[0].cb == p.nb);
      const bool cl = !(pcs[np - 1].ca == 0 && pcs[np - 1].cb == p.nb) && !(first && np == 1);
      if (c0) {
        cutA_ti = ti;
        cutA_g = pcs[0].g;
        if (ck == 0) crowA = crow;
      }
      if (cl) {
        cutB_ti = ti;
        cutB_g = pcs[np - 1].g;
        warpB = np - 1;
        if (ck == np - 1) crowB = crow;
      }
    }
    __syncthreads();
    first = false;
    u = uu;
  }
  if (cutA_ti >= 0 || cutB_ti >= 0) {
    // Each CTA publishes its partial sums of a cut row group and counts its
    // arrival; the CTA that arrives last adds the slots in CTA order and
    // writes y.  No CTA waits for another.  (The last round ended with a
    // barrier, so this CTA's slot writes precede the fence.)
    __shared__ int sflag[2];
    const int side = threadIdx.x == 0 ? 0 : threadIdx.x == 32 ? 1 : -1;
    if (side >= 0 && (side ? cutB_ti : cutA_ti) >= 0) {
      const TensorArgs &TX = tens[side ? cutB_ti : cutA_ti];
      const int64_t g = side ? cutB_g : cutA_g, gu = TX.ubegin + g * TX.p.nb;
      const int cf = cta_of(cb, a.ctas, gu), cl = cta_of(cb, a.ctas, gu + TX.p.nb - 1);
      __threadfence();
      const int old = atomicAdd(TX.p.counters + g, 1);
      const bool last = (old == cl - cf);
      if (last) __threadfence();
      sflag[side] = last ? 1 : 0;
    }
    __syncthreads();
#pragma unroll
    for (int side = 0; side < 2; ++side) {
      const int xti = side ? cutB_ti : cutA_ti;
      if (xti < 0 || warp != (side ? warpB : 0) || !sflag[side]) continue;
      const TensorArgs &TX = tens[xti];
      const int64_t g = side ? cutB_g : cutA_g, gu = TX.ubegin + g * TX.p.nb;
      const int cf = cta_of(cb, a.ctas, gu), cl = cta_of(cb, a.ctas, gu + TX.p.nb - 1);
      const int32_t rr = side ? crowB : crowA;
      float *y = kSet ? a.Yall + (int64_t)a.n * TX.rpre : TX.y;
      const uint16_t *x = kSet ? a.Xall + (int64_t)a.n * TX.cpre : TX.x;
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        float v = 0.f;
        for (int c2 = cf; c2 <= cl; ++c2) {
          const int s2 = (cb[c2] >= gu) ? 0 : 1;
          v += __ldcg(TX.p.slots + ((int64_t)c2 * 2 + s2) * 32 * kMaxBatch + lane * NB + b);
        }
        if (rr >= 0 && b < a.n) y[(int64_t)b * TX.p.R + rr] = v + outlier_term(TX.p, x, rr, b);
      }
      if (lane == 0) TX.p.counters[g] = 0;
    }
  }
}

// Activations in permuted column order, zero at outlier columns (their
// contribution is added exactly by the epilogue), weight-major with NB values
// per weight: xperm[p * NB + b] = x_b[perm[p]] (0 for b >= n).  One grid row
// per tensor.
struct XpermArgs {
  struct {
    const int32_t *perm;
    const uint16_t *x;
    float *xperm;
    int64_t C;
    int32_t n_out;
    int32_t out_cols[kMaxOutliers];
  } t[kMaxTensors];
  int n;   // batch columns
  int nbt; // batch template: values per weight in the scratch layout
};

__global__ void k_xperm(const __grid_constant__ XpermArgs a) {
  // The fused kernel may start launching now; it waits for this grid's writes.
  asm volatile("griddepcontrol.launch_dependents;");
  const auto &T = a.t[blockIdx.y];
  const int64_t total = (int64_t)a.nbt * T.C;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t pc = t / a.nbt;
    const int b = (int)(t - pc * a.nbt);
    float v = 0.f;
    if (b < a.n) {
      const int col = __ldg(T.perm + pc);
      bool outl = false;
      for (int o = 0; o < T.n_out; ++o) outl |= (T.out_cols[o] == col);
      v = outl ? 0.f : bf16_to_f32(__ldg(T.x + (int64_t)b * T.C + col));
    }
    T.xperm[t] = v;
  }
}

// The same for a layer set: descriptors in device memory, x of tensor i at
// Xall + n * cpre_i.
__global__ void k_xperm_set(const TensorArgs *__restrict__ tens, const uint16_t *Xall, int n, int nbt) {
  asm volatile("griddepcontrol.launch_dependents;");
  const TensorArgs &T = tens[blockIdx.y];
  const LayerArgs &p = T.p;
  const uint16_t *x = Xall + (int64_t)n * T.cpre;
  const int64_t total = (int64_t)nbt * p.C;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t pc = t / nbt;
    const int b = (int)(t - pc * nbt);
    float v = 0.f;
    if (b < n) {
      const int col = __ldg(p.perm + pc);
      bool outl = false;
      for (int o = 0; o < p.n_out; ++o) outl |= (p.out_cols[o] == col);
      v = outl ? 0.f : bf16_to_f32(__ldg(x + (int64_t)b * p.C + col));
    }
    p.xperm[t] = v;
  }
}

template <int NB>
static size_t smem_bytes() {
  return sizeof(uint64_t) * 512 * kTableSlots + (size_t)kWarps * Cfg<NB>::WARP_BYTES +
         sizeof(float) * Cfg<NB>::RG * kWarps * 32 * NB + sizeof(uint4) * Cfg<NB>::RG * 32 * 2;
}

// The fused kernel's dynamic shared-memory limit is a per-device attribute:
// set once per device (any host thread), and set again if a launch reports an
// invalid configuration (the device's context may have been reset since).
template <int NB, bool kSet>
static DeviceOnce &smem_once() {
  static DeviceOnce once;
  return once;
}

template <int NB, bool kSet>
static cudaError_t set_smem_limit(int dev) {
  return (cudaError_t)smem_once<NB, kSet>().run(dev, [] {
    return (int)cudaFuncSetAttribute(k_gemv<NB, kSet>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)smem_bytes<NB>());
  });
}

template <int NB, bool kSet>
static cudaError_t launch_fused(const cudaLaunchConfig_t &cfg, const MultiArgs &a) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = set_smem_limit<NB, kSet>(dev);
  if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, k_gemv<NB, kSet>, a);
  if (e == cudaErrorInvalidValue) {
    (void)cudaGetLastError();
    smem_once<NB, kSet>().forget(dev);
    e = set_smem_limit<NB, kSet>(dev);
    if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, k_gemv<NB, kSet>, a);
  }
  return e;
}

// Cost-balanced ranges of the units of all tensors, one per CTA.  A group's
// cost is its modeled time at batch n (block passes and the sum of k over
// them); inside the group where a range is cut, the first row's rung profile,
// scaled to the group's cost, places the cut.  One sweep over the groups
// places all cuts in order.
static void partition(const seedq_layer *const *layers, int nt, int n, int64_t *ubegin, int64_t *cta_begin,
                      int &ctas_out) {
  const double cb = cost_block(n);
  auto gcost = [&](const seedq_layer *L, int64_t g) { return kCostK * L->h_gk[g] + cb * L->h_gp[g]; };
  int64_t U = 0;
  double total = 0.0;
  for (int i = 0; i < nt; ++i) {
    const seedq_layer *L = layers[i];
    const int64_t G = (L->args.R + 31) / 32;
    ubegin[i] = U;
    U += G * L->args.nb;
    total += gcost(L, G);
  }
  int ctas = layers[0]->max_ctas;
  if (ctas > kMaxCtas) ctas = kMaxCtas;
  if (U < ctas) ctas = (int)U;
  ctas_out = ctas;
  cta_begin[0] = 0;
  cta_begin[ctas] = U;
  int c = 1;
  double tbase = 0.0;  // cost of the tensors before the current one
  for (int ti = 0; ti < nt && c < ctas; ++ti) {
    const seedq_layer *L = layers[ti];
    const int64_t G = (L->args.R + 31) / 32;
    const int J = L->args.J, Jm1 = J > 1 ? J - 1 : 1, nb = L->args.nb;
    for (int64_t g = 0; g < G && c < ctas; ++g) {
      const double g0 = gcost(L, g), g1 = gcost(L, g + 1);
      double target = total * c / ctas;
      if (target - tbase >= g1) continue;
      const int32_t *b = L->h_repbk + g * Jm1;
      double rep = 0.0;
      for (int j = 0, clo = 0; j < J; ++j) {
        const int chi = (j < J - 1) ? b[j] : nb;
        rep += (kCostK * L->k[j] + cb) * (chi - clo);
        clo = chi;
      }
      const double scale = rep > 0.0 ? (g1 - g0) / rep : 1.0;
      while (c < ctas && target - tbase < g1) {
        const double lt = target - tbase;
        double acc = g0;
        int col = nb, clo = 0;
        for (int j = 0; j < J; ++j) {
          const int chi = (j < J - 1) ? b[j] : nb;
          const double per = (kCostK * L->k[j] + cb) * scale;
          const double seg = per * (chi - clo);
          if (acc + seg > lt) {
            col = clo + (int)((lt - acc) / per);
            break;
          }
          acc += seg;
          clo = chi;
        }
        if (col < 0) col = 0;
        if (col > nb) col = nb;
        int64_t u = ubegin[ti] + g * nb + col;
        if (u <= cta_begin[c - 1]) u = cta_begin[c - 1] + 1;
        if (u > U - (ctas - c)) u = U - (ctas - c);
        cta_begin[c] = u;
        ++c;
        target = total * c / ctas;
      }
    }
    tbase += gcost(L, G);
  }
  // Cuts left over by rounding at the very end of the sequence.
  for (; c < ctas; ++c) {
    int64_t u = cta_begin[c - 1] + 1;
    if (u > U - (ctas - c)) u = U - (ctas - c);
    cta_begin[c] = u;
  }
}

template <int NB>
static seedq_status launch(const seedq_layer *const *layers, int nt, const uint16_t *const *x, int n,
                           float *const *y, cudaStream_t st) {
  MultiArgs args;
  MultiArgs *a = &args;
  a->nt = nt;
  a->n = n;
  a->zero = 0u;
  for (int i = 0; i < nt; ++i) {
    a->t[i].p = layers[i]->args;
    a->t[i].x = x[i];
    a->t[i].y = y[i];
    a->t[i].stream_bytes = layers[i]->stream_bytes;
  }
  int64_t ub[kMaxTensors];
  partition(layers, nt, n, ub, a->cta_begin, a->ctas);
  for (int i = 0; i < nt; ++i) a->t[i].ubegin = ub[i];
  a->tens = nullptr;
  a->cbd = nullptr;
  a->Xall = nullptr;
  a->Yall = nullptr;
  seedq_status rc = SEEDQ_OK;
  {
    XpermArgs xa;
    xa.n = n;
    xa.nbt = NB;
    int64_t maxC = 0;
    for (int i = 0; i < nt; ++i) {
      const LayerArgs &p = layers[i]->args;
      xa.t[i].perm = p.perm;
      xa.t[i].x = x[i];
      xa.t[i].xperm = p.xperm;
      xa.t[i].C = p.C;
      xa.t[i].n_out = p.n_out;
      for (int o = 0; o < kMaxOutliers; ++o) xa.t[i].out_cols[o] = p.out_cols[o];
      if (p.C > maxC) maxC = p.C;
    }
    const int64_t want = ((int64_t)NB * maxC + 255) / 256;
    const int gx = (int)(want < 64 ? want : 64);
    k_xperm<<<dim3(gx, nt), 256, 0, st>>>(xa);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) {
      // Programmatic dependent launch: the fused kernel's CTAs may start (and
      // stage their jump tables) while the pre-kernel finishes; they wait for
      // its writes before the first activation load.
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(a->ctas);
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = smem_bytes<NB>();
      cfg.stream = st;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[0].val.programmaticStreamSerializationAllowed = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      e = launch_fused<NB, false>(cfg, *a);
    }
    if (e != cudaSuccess) rc = cuda_fail(e);
  }
  return rc;
}

static seedq_status gemm_multi(const seedq_layer *const *layers, int nt, const uint16_t *const *X,
                               int n, float *const *Y, cudaStream_t st) {
  if (!layers || !X || !Y || nt < 1 || nt > kMaxTensors || n < 1 || n > kMaxBatch)
    return SEEDQ_ERR_INVALID_ARG;
  for (int i = 0; i < nt; ++i) {
    if (!layers[i] || !X[i] || !Y[i] || n > layers[i]->max_batch) return SEEDQ_ERR_INVALID_ARG;
    if (!layers[i]->args.stream) return SEEDQ_ERR_STREAM;
  }
  switch (batch_template(n)) {
    case 1: return launch<1>(layers, nt, X, n, Y, st);
    case 2: return launch<2>(layers, nt, X, n, Y, st);
    case 4: return launch<4>(layers, nt, X, n, Y, st);
    case 8: return launch<8>(layers, nt, X, n, Y, st);
    default: return launch<16>(layers, nt, X, n, Y, st);
  }
}

}  // namespace seedq

// Every tensor of a model (or any group of prepared layers) under one launch:
// descriptors and, per batch template, the cost-balanced CTA ranges live in
// device memory, built once when the set is created.
struct seedq_layer_set {
  int nt = 0;
  int max_batch = 0;
  int64_t cols = 0, rows = 0;            // totals: x holds n * cols values, y n * rows
  std::vector<int64_t> cpre, rpre;       // nt + 1 prefix sums
  seedq::TensorArgs *d_tens = nullptr;   // nt descriptors
  int64_t *d_cta[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};  // per batch template
  int ctas[5] = {0, 0, 0, 0, 0};
  int64_t maxC = 0;
};

namespace seedq {

static int tmpl_index(int nb) { return nb <= 1 ? 0 : nb <= 2 ? 1 : nb <= 4 ? 2 : nb <= 8 ? 3 : 4; }

template <int NB>
static seedq_status launch_set(const seedq_layer_set *S, const uint16_t *X, int n, float *Y,
                               cudaStream_t st) {
  MultiArgs a;
  memset(&a, 0, sizeof a);
  a.nt = S->nt;
  a.n = n;
  a.zero = 0u;
  a.ctas = S->ctas[tmpl_index(NB)];
  a.tens = S->d_tens;
  a.cbd = S->d_cta[tmpl_index(NB)];
  a.Xall = X;
  a.Yall = Y;
  const int64_t want = ((int64_t)NB * S->maxC + 255) / 256;
  const int gx = (int)(want < 64 ? want : 64);
  k_xperm_set<<<dim3(gx, S->nt), 256, 0, st>>>(S->d_tens, X, n, NB);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.ctas);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_bytes<NB>();
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = launch_fused<NB, true>(cfg, a);
  }
  return e == cudaSuccess ? SEEDQ_OK : cuda_fail(e);
}

static void free_set(seedq_layer_set *S) {
  if (!S) return;
  cudaFree(S->d_tens);
  for (int i = 0; i < 5; ++i) cudaFree(S->d_cta[i]);
  delete S;
}

}  // namespace seedq

using namespace seedq;

extern "C" {

seedq_status seedq_layer_set_create(const seedq_layer *const *layers, int32_t count,
                                    seedq_layer_set **out) {
  if (!layers || !out || count < 1 || count > 65535) return SEEDQ_ERR_INVALID_ARG;
  *out = nullptr;
  int mb = kMaxBatch;
  for (int i = 0; i < count; ++i) {
    if (!layers[i]) return SEEDQ_ERR_INVALID_ARG;
    if (!layers[i]->args.stream) return SEEDQ_ERR_STREAM;
    if (layers[i]->max_batch < mb) mb = layers[i]->max_batch;
  }
  seedq_layer_set *S = new (std::nothrow) seedq_layer_set;
  if (!S) return SEEDQ_ERR_NOMEM;
  S->nt = count;
  S->max_batch = mb;
  S->cpre.assign(count + 1, 0);
  S->rpre.assign(count + 1, 0);
  for (int i = 0; i < count; ++i) {
    S->cpre[i + 1] = S->cpre[i] + layers[i]->args.C;
    S->rpre[i + 1] = S->rpre[i] + layers[i]->args.R;
    if (layers[i]->args.C > S->maxC) S->maxC = layers[i]->args.C;
  }
  S->cols = S->cpre[count];
  S->rows = S->rpre[count];
  std::vector<TensorArgs> h(count);
  std::vector<int64_t> ub(count), cta(kMaxCtas + 1);
  seedq_status rc = SEEDQ_OK;
  cudaError_t e = cudaSuccess;
  for (int k = 0; k < 5 && rc == SEEDQ_OK && e == cudaSuccess; ++k) {
    const int nb = 1 << k;
    if (k > 0 && (1 << (k - 1)) >= mb) break;  // templates above max_batch are never launched
    int ctas = 0;
    partition(layers, count, nb, ub.data(), cta.data(), ctas);
    S->ctas[k] = ctas;
    e = cudaMalloc((void **)&S->d_cta[k], sizeof(int64_t) * (ctas + 1));
    if (e == cudaSuccess)
      e = cudaMemcpy(S->d_cta[k], cta.data(), sizeof(int64_t) * (ctas + 1), cudaMemcpyHostToDevice);
  }
  for (int i = 0; i < count; ++i) {
    memset(&h[i], 0, sizeof(TensorArgs));
    h[i].p = layers[i]->args;
    h[i].ubegin = ub[i];
    h[i].stream_bytes = layers[i]->stream_bytes;
    h[i].cpre = S->cpre[i];
    h[i].rpre = S->rpre[i];
  }
  if (e == cudaSuccess) e = cudaMalloc((void **)&S->d_tens, sizeof(TensorArgs) * count);
  if (e == cudaSuccess)
    e = cudaMemcpy(S->d_tens, h.data(), sizeof(TensorArgs) * count, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) rc = cuda_fail(e);
  if (rc != SEEDQ_OK) {
    free_set(S);
    return rc;
  }
  *out = S;
  return SEEDQ_OK;
}

seedq_status seedq_layer_set_layout(const seedq_layer_set *S, int64_t *col_offsets,
                                    int64_t *row_offsets) {
  if (!S) return SEEDQ_ERR_INVALID_ARG;
  for (int i = 0; i <= S->nt; ++i) {
    if (col_offsets) col_offsets[i] = S->cpre[i];
    if (row_offsets) row_offsets[i] = S->rpre[i];
  }
  return SEEDQ_OK;
}

seedq_status seedq_gemm_set(const seedq_layer_set *S, const uint16_t *X, int32_t n, float *Y,
                            void *cuda_stream) {
  if (!S || !X || !Y || n < 1 || n > S->max_batch) return SEEDQ_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  switch (batch_template(n)) {
    case 1: return launch_set<1>(S, X, n, Y, st);
    case 2: return launch_set<2>(S, X, n, Y, st);
    case 4: return launch_set<4>(S, X, n, Y, st);
    case 8: return launch_set<8>(S, X, n, Y, st);
    default: return launch_set<16>(S, X, n, Y, st);
  }
}

seedq_status seedq_layer_set_release(seedq_layer_set *S) {
  if (!S) return SEEDQ_ERR_INVALID_ARG;
  free_set(S);
  return SEEDQ_OK;
}

seedq_status seedq_gemm_small_batch(const seedq_layer *L, const uint16_t *X, int32_t n, float *Y,
                                    void *cuda_stream) {
  return gemm_multi(&L, 1, &X, n, &Y, (cudaStream_t)cuda_stream);
}

seedq_status seedq_gemv(const seedq_layer *L, const uint16_t *x, float *y, void *cuda_stream) {
  return gemm_multi(&L, 1, &x, 1, &y, (cudaStream_t)cuda_stream);
}

seedq_status seedq_gemm_multi(const seedq_layer *const *layers, int32_t count,
                              const uint16_t *const *X, int32_t n, float *const *Y,
                              void *cuda_stream) {
  return gemm_multi(layers, count, X, n, Y, (cudaStream_t)cuda_stream);
}

}  // extern "C"
