// Fused reconstruction x matrix-vector product: y = W_hat x and the decode-batch
// skinny GEMM Y = X W_hat^T (n <= 16).  W_hat is never written to memory; HBM
// carries only the compressed stream, the plan rows and x / y.
#include <cuda_fp16.h>

#include "seedq_internal.cuh"

namespace seedq {

constexpr int kThreads = 256;           // 8 warps
constexpr int kWarps = kThreads / 32;
constexpr int kXFloats = 8192;          // 32 KB of staged activations per CTA

// Column blocks per split for batch n: the activation slice of a split
// (n x 8 cb floats, permuted order) fills the 32 KB staging buffer.
__host__ __device__ inline int cb_for(int n) { return kXFloats / 8 / n; }

// Batch sizes run by one of the instantiated kernels: 1, 2, 4, 8, 16.
__host__ __device__ inline int batch_template(int n) {
  return n <= 1 ? 1 : n <= 2 ? 2 : n <= 4 ? 4 : n <= 8 ? 8 : 16;
}

// Split-K partial sums the layer must hold for batches up to max_batch.
int64_t gemv_partial_elems(const seedq_layer *L, int max_batch) {
  int64_t need = 0;
  for (int nt = 1; nt <= batch_template(max_batch); nt *= 2) {
    const int cb = cb_for(nt);
    const int64_t ns = (L->args.nb + cb - 1) / cb;
    const int64_t e = ns > 1 ? ns * (nt < max_batch ? nt : max_batch) * L->args.R : 0;
    if (e > need) need = e;
  }
  return need;
}

struct GemvArgs {
  LayerArgs p;
  const uint16_t *x;  // n x C bf16, original column order
  float *y;           // n x R
  float *partials;    // nsplit x n x R
  int n;
  int cb;
  int nsplit;
  int64_t nrt;        // row tiles (kWarps rows each)
  int64_t ntiles;
};

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }

// One block of rung (S,K): reconstruct exactly, then acc[b] += scale * sum_i I_i x_b,i.
template <int S, int K, int NB>
__device__ __forceinline__ void gemv_block(const LayerArgs &p, uint64_t off, const uint64_t *tab,
                                           const float *xc, int xstride, float (&acc)[NB]) {
  uint32_t lo, hi;
  load_bits<RungT<S, K>::NWORDS>(p.stream, off, lo, hi);
  float I[8], scale;
  reconstruct<S, K>(lo, hi, tab, I, scale);
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const float4 x0 = *reinterpret_cast<const float4 *>(xc + b * xstride);
    const float4 x1 = *reinterpret_cast<const float4 *>(xc + b * xstride + 4);
    float s = I[0] * x0.x;
    s = __fmaf_rn(I[1], x0.y, s);
    s = __fmaf_rn(I[2], x0.z, s);
    s = __fmaf_rn(I[3], x0.w, s);
    s = __fmaf_rn(I[4], x1.x, s);
    s = __fmaf_rn(I[5], x1.y, s);
    s = __fmaf_rn(I[6], x1.z, s);
    s = __fmaf_rn(I[7], x1.w, s);
    acc[b] = __fmaf_rn(scale, s, acc[b]);
  }
}

template <int NB>
__device__ __forceinline__ void dispatch_block(int code, const LayerArgs &p, uint64_t off,
                                               const uint64_t *tab, const float *xc, int xstride,
                                               float (&acc)[NB]) {
  switch (code) {
#define SEEDQ_CASE(S_, K_)                                      \
  case rung_code(S_, K_):                                       \
    gemv_block<S_, K_, NB>(p, off, tab, xc, xstride, acc);      \
    break;
    SEEDQ_FOR_EACH_RUNG(SEEDQ_CASE)
#undef SEEDQ_CASE
    default:
      break;
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

// One warp, one row, one column split [cb0, cb1): lanes take consecutive blocks.
// Rungs are non-decreasing along a row, so almost every group of 32 blocks has a
// single rung: then lane offsets are base + lane * l(g), and the rung dispatch
// is warp-uniform.  Groups that straddle a breakpoint run once per rung present.
template <int NB>
__device__ void gemv_row(const GemvArgs &a, const uint64_t *tabs, const float *xs, int64_t r,
                         int s, int cb0, int cb1, int lane) {
  const LayerArgs &p = a.p;
  const int J = p.J;
  int32_t bk[kMaxJ];
#pragma unroll
  for (int j = 0; j < kMaxJ - 1; ++j) bk[j] = (j < J - 1) ? __ldg(p.brk + r * (J - 1) + j) : p.nb;
  uint64_t off = __ldg(p.row_off + r) + bits_before(bk, J, p.L, p.nb, cb0);
  const int xstride = a.cb * 8;
  float acc[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) acc[b] = 0.f;
  int seg = rung_of(bk, J, cb0);
  for (int g0 = cb0; g0 < cb1; g0 += 32) {
    const int gend = min(g0 + 32, cb1);
    while (seg < J - 1 && bk[seg] <= g0) ++seg;
    const int c = g0 + lane;
    const bool valid = c < gend;
    const float *xc = xs + (c - cb0) * 8;
    const int seg_end = (seg < J - 1) ? bk[seg] : p.nb;
    if (seg_end >= gend) {
      const int Lg = p.L[seg];
      if (valid)
        dispatch_block<NB>(p.code[seg], p, off + (uint64_t)lane * Lg,
                           tabs + p.slot[seg] * 512, xc, xstride, acc);
      off += (uint64_t)(gend - g0) * Lg;
    } else {
      const int myr = rung_of(bk, J, c);
      const uint64_t base = bits_before(bk, J, p.L, p.nb, g0);
      const uint64_t myoff = off + (bits_before(bk, J, p.L, p.nb, c) - base);
      const int last = rung_of(bk, J, gend - 1);
      for (int rr = seg; rr <= last; ++rr)
        if (valid && myr == rr)
          dispatch_block<NB>(p.code[rr], p, myoff, tabs + p.slot[rr] * 512, xc, xstride, acc);
      off += bits_before(bk, J, p.L, p.nb, gend) - base;
    }
  }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    float v = acc[b];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    acc[b] = v;
  }
  if (lane == 0) {
    for (int b = 0; b < a.n && b < NB; ++b) {
      if (a.nsplit == 1) a.y[(int64_t)b * p.R + r] = acc[b] + outlier_term(a, r, b);
      else a.partials[((int64_t)s * a.n + b) * p.R + r] = acc[b];
    }
  }
}

template <int NB>
__global__ void __launch_bounds__(kThreads) k_gemv(const __grid_constant__ GemvArgs a) {
  extern __shared__ __align__(16) uint64_t smem[];
  const LayerArgs &p = a.p;
  uint64_t *tabs = smem;
  float *xs = reinterpret_cast<float *>(smem + p.nslots * 512);
  for (int i = threadIdx.x; i < p.nslots * 512; i += kThreads) tabs[i] = __ldg(p.tables + i);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int cur_s = -1;
  for (int64_t t = blockIdx.x; t < a.ntiles; t += gridDim.x) {
    const int s = (int)(t / a.nrt);
    const int64_t rt = t - (int64_t)s * a.nrt;
    const int cb0 = s * a.cb, cb1 = min(cb0 + a.cb, p.nb);
    if (s != cur_s) {
      __syncthreads();
      const int span = a.cb * 8, ncols = (cb1 - cb0) * 8;
      for (int idx = threadIdx.x; idx < NB * span; idx += kThreads) {
        const int b = idx / span, pc = idx - b * span;
        float v = 0.f;
        if (b < a.n && pc < ncols) {
          const int col = __ldg(p.perm + cb0 * 8 + pc);
          bool outl = false;
          for (int o = 0; o < p.n_out; ++o) outl |= (p.out_cols[o] == col);
          if (!outl) v = bf16_to_f32(a.x[(int64_t)b * p.C + col]);
        }
        xs[idx] = v;
      }
      __syncthreads();
      cur_s = s;
    }
    const int64_t r = rt * kWarps + warp;
    if (r < p.R) gemv_row<NB>(a, tabs, xs, r, s, cb0, cb1, lane);
  }
}

// Deterministic split-K reduction (splits summed in ascending order) + outliers.
__global__ void k_reduce(const __grid_constant__ GemvArgs a) {
  const int64_t total = (int64_t)a.n * a.p.R;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int b = (int)(t / a.p.R);
    const int64_t r = t - (int64_t)b * a.p.R;
    float v = 0.f;
    for (int s = 0; s < a.nsplit; ++s) v += a.partials[((int64_t)s * a.n + b) * a.p.R + r];
    a.y[t] = v + outlier_term(a, r, b);
  }
}

template <int NB>
static seedq_status launch(const seedq_layer *L, const uint16_t *x, int n, float *y,
                           cudaStream_t st) {
  GemvArgs a;
  a.p = L->args;
  a.x = x;
  a.y = y;
  a.partials = L->d_partials;
  a.n = n;
  a.cb = cb_for(NB);
  a.nsplit = (L->args.nb + a.cb - 1) / a.cb;
  a.nrt = (L->args.R + kWarps - 1) / kWarps;
  a.ntiles = a.nrt * a.nsplit;
  if (a.nsplit > 1 && (int64_t)a.nsplit * n * L->args.R > L->partial_elems) return SEEDQ_ERR_INVALID_ARG;
  const size_t smem = sizeof(uint64_t) * 512 * L->args.nslots + sizeof(float) * NB * a.cb * 8;
  static bool attr_set = false;
  if (!attr_set) {
    SEEDQ_CUDA(cudaFuncSetAttribute(k_gemv<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)(sizeof(uint64_t) * 512 * kMaxJ + sizeof(float) * kXFloats)));
    attr_set = true;
  }
  int dev = 0, sms = 0, occ = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  SEEDQ_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_gemv<NB>, kThreads, smem));
  if (occ < 1) occ = 1;
  const int64_t want = (int64_t)sms * occ;
  const int grid = (int)(a.ntiles < want ? a.ntiles : want);
  k_gemv<NB><<<grid, kThreads, smem, st>>>(a);
  SEEDQ_CUDA(cudaGetLastError());
  if (a.nsplit > 1) {
    const int64_t total = (int64_t)n * L->args.R;
    const int g = (int)((total + 255) / 256 < (int64_t)sms * 8 ? (total + 255) / 256 : (int64_t)sms * 8);
    k_reduce<<<g, 256, 0, st>>>(a);
    SEEDQ_CUDA(cudaGetLastError());
  }
  return SEEDQ_OK;
}

}  // namespace seedq

using namespace seedq;

extern "C" {

seedq_status seedq_gemm_small_batch(const seedq_layer *L, const uint16_t *X, int32_t n, float *Y,
                                    void *cuda_stream) {
  if (!L || !X || !Y || n < 1 || n > L->max_batch) return SEEDQ_ERR_INVALID_ARG;
  if (!L->args.stream) return SEEDQ_ERR_STREAM;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  if (n == 1) return launch<1>(L, X, n, Y, st);
  if (n == 2) return launch<2>(L, X, n, Y, st);
  if (n <= 4) return launch<4>(L, X, n, Y, st);
  if (n <= 8) return launch<8>(L, X, n, Y, st);
  return launch<16>(L, X, n, Y, st);
}

seedq_status seedq_gemv(const seedq_layer *L, const uint16_t *x, float *y, void *cuda_stream) {
  if (!L || !x || !y) return SEEDQ_ERR_INVALID_ARG;
  if (!L->args.stream) return SEEDQ_ERR_STREAM;
  return launch<1>(L, x, 1, y, (cudaStream_t)cuda_stream);
}

}  // extern "C"
