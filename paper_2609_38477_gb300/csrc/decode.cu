// Alg. 2 in full: materialize W_hat (rows of it) in the original column order.
#include <cuda_fp16.h>

#include "seedq_internal.cuh"

namespace seedq {

template <int K>
__device__ __forceinline__ void decode_block(const LayerArgs &p, int S, uint64_t off,
                                             const uint64_t *tab, float *Wrow, int c) {
  uint32_t lo, hi;
  load_bits<3>(p.stream, off, lo, hi);  // the stream buffer ends in 16 bytes of slack
  float I[8], scale;
  const RungRt<K> rc(S, p.zero);
  reconstruct_rt<K>(lo, hi, tab, rc, I, scale);
#pragma unroll
  for (int i = 0; i < 8; ++i) Wrow[__ldg(p.perm + 8 * c + i)] = I[i] * scale;  // exact
}

// One thread per block; reads l(g_b) bits at the block's offset (row offset +
// closed form over the row's rung breakpoints), writes 8 weights through the
// inverse permutation (the scatter step of Alg. 2).
__global__ void __launch_bounds__(256) k_decode(const __grid_constant__ LayerArgs p, int64_t row0, int64_t nrows, float *W) {
  const int64_t total = nrows * (int64_t)p.nb;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < total;
       b += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = b / p.nb;
    const int c = (int)(b - i * p.nb);
    const int64_t r = row0 + i;
    int32_t bk[kMaxJ];
    for (int j = 0; j < p.J - 1; ++j) bk[j] = __ldg(p.brk + r * (p.J - 1) + j);
    const int g = rung_of(bk, p.J, c);
    const uint64_t roff = __ldg(p.row_off + r);
    const uint64_t off = roff + bits_before(bk, p.J, p.L, p.nb, c);
    // The plan and the bound buffer must agree: the last block of a row ends
    // at the next row's offset, and the block's three words are readable.
    // Otherwise flag bit 0 and leave the block's weights unwritten.
    if (c == p.nb - 1 && off + (uint64_t)p.L[g] != __ldg(p.row_off + r + 1)) atomicOr(p.flags, 1u);
    if ((off >> 5) + 3 > p.stream_words) {
      atomicOr(p.flags, 1u);
      continue;
    }
    const uint64_t *tab = p.tables + (size_t)p.slot[g] * 512;
    float *Wrow = W + i * p.C;
    const int S = rung_S(p.code[g]);
    switch (rung_K(p.code[g])) {
      case 2: decode_block<2>(p, S, off, tab, Wrow, c); break;
      case 3: decode_block<3>(p, S, off, tab, Wrow, c); break;
      case 4: decode_block<4>(p, S, off, tab, Wrow, c); break;
      case 5: decode_block<5>(p, S, off, tab, Wrow, c); break;
      case 6: decode_block<6>(p, S, off, tab, Wrow, c); break;
      default: atomicOr(p.flags, 1u);
    }
  }
}

// Outlier columns overwrite the codec's values (Alg. 2 last step; Sec. 3.5).
__global__ void k_outliers(const __grid_constant__ LayerArgs p, int64_t row0, int64_t nrows, float *W) {
  const int64_t total = nrows * p.n_out;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = t / p.n_out;
    const int o = (int)(t - i * p.n_out);
    const uint16_t h = p.out_vals[(row0 + i) * p.n_out + o];
    W[i * p.C + p.out_cols[o]] = __half2float(__ushort_as_half(h));
  }
}

}  // namespace seedq

using namespace seedq;

extern "C" {

seedq_status seedq_decode_rows(const seedq_layer *L, int64_t row0, int64_t nrows, float *W,
                               void *cuda_stream) {
  if (!L || !W || row0 < 0 || nrows < 0 || row0 + nrows > L->args.R) return SEEDQ_ERR_INVALID_ARG;
  if (!L->args.stream) return SEEDQ_ERR_STREAM;
  if (nrows == 0) return SEEDQ_OK;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t blocks = nrows * (int64_t)L->args.nb;
  const int64_t want = (blocks + 255) / 256;
  const int grid = (int)(want < (int64_t)sms * 16 ? want : (int64_t)sms * 16);
  k_decode<<<grid, 256, 0, st>>>(L->args, row0, nrows, W);
  SEEDQ_CUDA(cudaGetLastError());
  if (L->args.n_out > 0) {
    const int64_t t = nrows * L->args.n_out;
    const int g2 = (int)((t + 255) / 256 < 4096 ? (t + 255) / 256 : 4096);
    k_outliers<<<g2, 256, 0, st>>>(L->args, row0, nrows, W);
    SEEDQ_CUDA(cudaGetLastError());
  }
  return SEEDQ_OK;
}

seedq_status seedq_decode_weights(const seedq_layer *L, float *W, void *cuda_stream) {
  if (!L) return SEEDQ_ERR_INVALID_ARG;
  return seedq_decode_rows(L, 0, L->args.R, W, cuda_stream);
}

}  // extern "C"
