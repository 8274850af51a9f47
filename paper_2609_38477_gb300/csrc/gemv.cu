// Fused reconstruction x matrix-vector product: y = W_hat x, and the decode-batch
// skinny GEMM Y = X W_hat^T (n <= 16).  W_hat is never written to memory; HBM
// carries only the compressed stream, the plan rows and x / y.
//
// Work layout: a persistent kernel, one 24-warp CTA per SM.  A CTA owns a
// contiguous range of rows (a row tile) and stages, once, the LFSR jump tables
// and the activations in permuted column order (all columns when they fit,
// else column chunks).  Within a tile and chunk, the row-major sequence of
// (row, block) pairs is cut into 24 equal contiguous ranges, one per warp, so
// every warp gets the same number of blocks whatever the row length.  Rows cut
// by a range boundary leave per-warp partial sums in shared memory that are
// added in warp order, so results are deterministic.
#include <cuda_fp16.h>

#include "seedq_internal.cuh"

namespace seedq {

constexpr int kWarps = 24;
constexpr int kThreads = kWarps * 32;
constexpr int kXBytes = 112 * 1024;     // staged activations per CTA
constexpr int kAccFloats = 8192;        // row-tile accumulators per CTA (rows x n)

struct GemvArgs {
  LayerArgs p;
  const uint16_t *x;  // n x C bf16, original column order
  float *y;           // n x R
  int n;
  int cw;             // column blocks per chunk
  int nchunks;
  int rt;             // rows per tile
  int ntiles;
  uint32_t zero;      // 0 at run time; keeps per-rung constants in registers
};

__host__ __device__ inline int batch_template(int n) {
  return n <= 1 ? 1 : n <= 2 ? 2 : n <= 4 ? 4 : n <= 8 ? 8 : 16;
}

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }

template <int S, int K, int NB>
__device__ __forceinline__ void block_fma(const uint32_t (&w)[3], uint32_t sh, const uint64_t *tab,
                                          const RungConsts<S, K> &rc, const float *xc,
                                          int xstride, float (&acc)[NB]) {
  const uint32_t lo = __funnelshift_r(w[0], w[1], sh);
  const uint32_t hi = __funnelshift_r(w[1], w[2], sh);
  float I[8], scale;
  reconstruct<S, K>(lo, hi, tab, rc, I, scale);
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const float4 x0 = *reinterpret_cast<const float4 *>(xc + b * xstride);
    const float4 x1 = *reinterpret_cast<const float4 *>(xc + b * xstride + 4);
    float sacc = I[0] * x0.x;
    sacc = __fmaf_rn(I[1], x0.y, sacc);
    sacc = __fmaf_rn(I[2], x0.z, sacc);
    sacc = __fmaf_rn(I[3], x0.w, sacc);
    sacc = __fmaf_rn(I[4], x1.x, sacc);
    sacc = __fmaf_rn(I[5], x1.y, sacc);
    sacc = __fmaf_rn(I[6], x1.z, sacc);
    sacc = __fmaf_rn(I[7], x1.w, sacc);
    acc[b] = __fmaf_rn(scale, sacc, acc[b]);
  }
}

// Blocks [s0, s0 + nblk) of one row, all at rung (S,K).  Lanes take
// consecutive blocks; 32 consecutive blocks span exactly L words, so each
// lane's in-word shift is fixed and its word pointer steps by L.  Words are
// loaded one group ahead.  xc0 points at the staged activations of block s0.
template <int S, int K, int NB>
__device__ __forceinline__ void run_segment(const uint32_t *__restrict__ base, uint32_t bit0,
                                            int nblk, const uint64_t *tab, const float *xc0,
                                            int xstride, int lane, uint32_t z, float (&acc)[NB]) {
  constexpr int L = RungT<S, K>::L;
  constexpr int NW = RungT<S, K>::NWORDS;
  const RungConsts<S, K> rc(z);
  const uint32_t b0 = bit0 + (uint32_t)lane * L;
  const uint32_t sh = b0 & 31;
  const uint32_t *q = base + (b0 >> 5);
  const float *xc = xc0 + lane * 8;
  const int ngroups = (nblk + 31) >> 5;
  int left = nblk - lane;  // blocks from this lane's current one to the segment end
  uint32_t w[3] = {0u, 0u, 0u};
  if (left > 0) {
#pragma unroll
    for (int i = 0; i < NW; ++i) w[i] = __ldg(q + i);
  }
  for (int g = 0; g < ngroups; ++g) {
    const uint32_t cur[3] = {w[0], w[1], w[2]};
    const bool mine = left > 0;
    left -= 32;
    q += L;
    if (left > 0) {
#pragma unroll
      for (int i = 0; i < NW; ++i) w[i] = __ldg(q + i);
    }
    if (mine) block_fma<S, K, NB>(cur, sh, tab, rc, xc, xstride, acc);
    xc += 256;
  }
}

// Blocks [ca, cb) of row r (a column range inside the staged chunk starting at
// block cb0).  Rungs are non-decreasing along a row, so the range crosses at
// most J rung segments; each runs a loop specialized for its rung.  Returns
// the warp-wide sums in acc (every lane holds them).
template <int NB>
__device__ __forceinline__ void row_range(const GemvArgs &a, const uint64_t *tabs, const float *xs,
                                          int64_t r, int ca, int cb, int cb0, int lane,
                                          float (&acc)[NB]) {
  const LayerArgs &p = a.p;
  const int J = p.J;
  const uint64_t roff = __ldg(p.row_off + r);
  const uint32_t *base = p.stream + (roff >> 5);
  const uint32_t rbit = (uint32_t)(roff & 31);
  const int xstride = a.cw * 8;
#pragma unroll
  for (int b = 0; b < NB; ++b) acc[b] = 0.f;
  uint32_t seg_bits = 0;  // bits of the row before block `lo`
  int lo = 0;
  for (int j = 0; j < J && lo < cb; ++j) {
    const int hi = (j < J - 1) ? __ldg(p.brk + r * (J - 1) + j) : p.nb;
    const int Lj = p.L[j];
    const int s0 = max(lo, ca), s1 = min(hi, cb);
    if (s0 < s1) {
      const uint32_t bit0 = rbit + seg_bits + (uint32_t)(s0 - lo) * Lj;
      const uint64_t *tab = tabs + p.slot[j] * 512;
      const float *xc0 = xs + (s0 - cb0) * 8;
      switch (p.code[j]) {
#define SEEDQ_CASE(S_, K_)                                                                  \
  case rung_code(S_, K_):                                                                   \
    run_segment<S_, K_, NB>(base, bit0, s1 - s0, tab, xc0, xstride, lane, a.zero, acc);     \
    break;
        SEEDQ_FOR_EACH_RUNG(SEEDQ_CASE)
#undef SEEDQ_CASE
        default:
          break;
      }
    }
    seg_bits += (uint32_t)(hi - lo) * Lj;
    lo = hi;
  }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    float v = acc[b];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    acc[b] = v;
  }
}

// Outlier epilogue: y_b[r] += sum_o W16[r, col_o] x_b[col_o] (Sec. 3.5).
__device__ __forceinline__ float outlier_term(const GemvArgs &a, int64_t r, int b) {
  float s = 0.f;
  for (int o = 0; o < a.p.n_out; ++o) {
    const float w = __half2float(__ushort_as_half(a.p.out_vals[r * a.p.n_out + o]));
    s = __fmaf_rn(w, bf16_to_f32(a.x[(int64_t)b * a.p.C + a.p.out_cols[o]]), s);
  }
  return s;
}

template <int NB>
__global__ void __launch_bounds__(kThreads, 1) k_gemv(const __grid_constant__ GemvArgs a) {
  extern __shared__ __align__(16) uint64_t smem[];
  const LayerArgs &p = a.p;
  uint64_t *tabs = smem;
  float *xs = reinterpret_cast<float *>(smem + p.nslots * 512);
  float *racc = xs + NB * a.cw * 8;               // rt x NB row accumulators
  float *slot = racc + a.rt * NB;                 // kWarps x 2 x NB partial sums
  int *slot_row = reinterpret_cast<int *>(slot + kWarps * 2 * NB);
  {
    const uint4 *src = reinterpret_cast<const uint4 *>(p.tables);
    uint4 *dst = reinterpret_cast<uint4 *>(tabs);
    for (int i = threadIdx.x; i < p.nslots * 256; i += kThreads) dst[i] = __ldg(src + i);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int tile = blockIdx.x; tile < a.ntiles; tile += gridDim.x) {
    const int64_t r_lo = (int64_t)tile * a.rt;
    const int nr = (int)min((int64_t)a.rt, p.R - r_lo);
    for (int i = threadIdx.x; i < nr * NB; i += kThreads) racc[i] = 0.f;
    for (int ch = 0; ch < a.nchunks; ++ch) {
      const int cb0 = ch * a.cw, cb1 = min(cb0 + a.cw, p.nb), ncb = cb1 - cb0;
      __syncthreads();
      // Stage the chunk's activations in permuted order (0 at outlier columns):
      // coalesced reads of x and of the inverse permutation, scattered into
      // shared memory, so no load waits on another.
      for (int col0 = threadIdx.x; col0 < p.C; col0 += 4 * kThreads) {
        int pos[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int col = col0 + u * kThreads;
          pos[u] = (col < p.C) ? __ldg(p.invperm + col) - cb0 * 8 : -1;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int col = col0 + u * kThreads;
          if (pos[u] >= 0 && pos[u] < ncb * 8) {
            bool outl = false;
            for (int o = 0; o < p.n_out; ++o) outl |= (p.out_cols[o] == col);
            for (int b = 0; b < a.n; ++b)
              xs[b * a.cw * 8 + pos[u]] = outl ? 0.f : bf16_to_f32(__ldg(a.x + (int64_t)b * p.C + col));
          }
        }
      }
      if (threadIdx.x < kWarps * 2) slot_row[threadIdx.x] = -1;
      __syncthreads();
      // This warp's equal share of the tile's (row, block) pairs in the chunk.
      const int64_t work = (int64_t)nr * ncb;
      const int64_t wb0 = work * warp / kWarps, wb1 = work * (warp + 1) / kWarps;
      int64_t wb = wb0;
      while (wb < wb1) {
        const int rr = (int)(wb / ncb);
        const int c0 = (int)(wb - (int64_t)rr * ncb);
        const int c1 = (int)min((int64_t)ncb, c0 + (wb1 - wb));
        float acc[NB];
        row_range<NB>(a, tabs, xs, r_lo + rr, cb0 + c0, cb0 + c1, cb0, lane, acc);
        if (lane == 0) {
          if (c0 == 0 && c1 == ncb) {  // whole row of the chunk: sole writer
#pragma unroll
            for (int b = 0; b < NB; ++b) racc[rr * NB + b] += acc[b];
          } else {
            const int s = (wb == wb0) ? 0 : 1;
            slot_row[warp * 2 + s] = rr;
#pragma unroll
            for (int b = 0; b < NB; ++b) slot[(warp * 2 + s) * NB + b] = acc[b];
          }
        }
        wb += c1 - c0;
      }
      __syncthreads();
      // Rows cut by range boundaries: add the partial sums in warp order.
      for (int rr = threadIdx.x; rr < nr; rr += kThreads) {
        for (int sidx = 0; sidx < kWarps * 2; ++sidx) {
          if (slot_row[sidx] == rr) {
            for (int b = 0; b < NB; ++b) racc[rr * NB + b] += slot[sidx * NB + b];
          }
        }
      }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nr * a.n; i += kThreads) {
      const int rr = i / a.n, b = i - rr * a.n;
      const int64_t r = r_lo + rr;
      a.y[(int64_t)b * p.R + r] = racc[rr * NB + b] + outlier_term(a, r, b);
    }
    __syncthreads();
  }
}

template <int NB>
static size_t smem_bytes(int nslots, int cw, int rt) {
  return sizeof(uint64_t) * 512 * nslots + sizeof(float) * NB * cw * 8 + sizeof(float) * rt * NB +
         sizeof(float) * kWarps * 2 * NB + sizeof(int) * kWarps * 2;
}

template <int NB>
static seedq_status launch(const seedq_layer *L, const uint16_t *x, int n, float *y,
                           cudaStream_t st) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  GemvArgs a;
  a.p = L->args;
  a.x = x;
  a.y = y;
  a.n = n;
  a.zero = 0u;
  const int cw_max = kXBytes / (int)sizeof(float) / 8 / NB;
  a.cw = L->args.nb < cw_max ? L->args.nb : cw_max;
  a.nchunks = (L->args.nb + a.cw - 1) / a.cw;
  int64_t rt = (L->args.R + sms - 1) / sms;
  if (rt * NB > kAccFloats) rt = kAccFloats / NB;
  a.rt = (int)rt;
  a.ntiles = (int)((L->args.R + rt - 1) / rt);
  const size_t smem = smem_bytes<NB>(L->args.nslots, a.cw, a.rt);
  static bool attr_set = false;
  if (!attr_set) {
    SEEDQ_CUDA(cudaFuncSetAttribute(k_gemv<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)smem_bytes<NB>(kMaxJ, cw_max, kAccFloats / NB)));
    attr_set = true;
  }
  const int grid = a.ntiles < sms ? a.ntiles : sms;
  k_gemv<NB><<<grid, kThreads, smem, st>>>(a);
  SEEDQ_CUDA(cudaGetLastError());
  return SEEDQ_OK;
}

// The fused kernel keeps no global scratch (partial sums live in shared memory).
int64_t gemv_partial_elems(const seedq_layer *, int) { return 0; }

}  // namespace seedq

using namespace seedq;

extern "C" {

seedq_status seedq_gemm_small_batch(const seedq_layer *L, const uint16_t *X, int32_t n, float *Y,
                                    void *cuda_stream) {
  if (!L || !X || !Y || n < 1 || n > L->max_batch) return SEEDQ_ERR_INVALID_ARG;
  if (!L->args.stream) return SEEDQ_ERR_STREAM;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  switch (batch_template(n)) {
    case 1: return launch<1>(L, X, n, Y, st);
    case 2: return launch<2>(L, X, n, Y, st);
    case 4: return launch<4>(L, X, n, Y, st);
    case 8: return launch<8>(L, X, n, Y, st);
    default: return launch<16>(L, X, n, Y, st);
  }
}

seedq_status seedq_gemv(const seedq_layer *L, const uint16_t *x, float *y, void *cuda_stream) {
  if (!L || !x || !y) return SEEDQ_ERR_INVALID_ARG;
  if (!L->args.stream) return SEEDQ_ERR_STREAM;
  return launch<1>(L, x, 1, y, (cudaStream_t)cuda_stream);
}

}  // extern "C"
