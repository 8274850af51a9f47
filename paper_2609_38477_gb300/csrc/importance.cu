// Data-free importance (Sec. 3.2, Eq. gamma, Eq. prop, the backward proxy of
// App. A.1) and the outlier-column statistics and selection (Sec. 3.5,
// App. A.6) over an FP16 checkpoint resident on the device.
//
// Every weight matrix is read once, by one column pass that computes for each
// tile of 32 input columns:
//   * the weighted column sums of squares sum_r W_rc^2 g_r of the backward
//     proxy (g the residual-gradient scale the matrix writes to),
//   * the partial row sums of squares sum_{c in tile} W_rc^2 a_c of Eq. prop
//     (for W_v, W_gate, W_up),
//   * the column maximum of |W| and a count that decides, exactly, which
//     columns can reach the dynamic-range threshold; those (in practice only
//     spiked columns) get their exact median from two more sweeps.
// Layers are taken in reverse order because each layer's column sums need the
// stream scale left by the layer above; a small kernel per step finishes the
// stream update, rho, a^(down) (Gauss-Hermite) and a^(o) (repeat_kv).
//
// Work distribution: persistent CTAs (two per SM) take (row slab, tile) items
// round-robin; each thread streams its own 16-byte pieces of 8 rows per stage
// through a three-stage cp.async ring in shared memory, so loads stay in
// flight across item boundaries; the last slab of a tile to finish combines
// the slabs' partial results in slab order.
//
// Arithmetic: squares of FP16 values are exact in fp32; each product with the
// fp32-rounded weight is rounded once, 16 rows accumulate in fp32 and then in
// fp64 (relative error of a column sum below 18 u, u = 2^-24, all terms being
// non-negative), partial row sums of 32 columns are fp32 and their tile sums
// compensated float32 sums; the stream scale stays fp64.  Tables are rounded to float32 (App.
// A.7).  The outlier statistics are exact: maxima and medians are FP16 values,
// the statistic is one IEEE division of their fp64 sum, and the activation
// mean is the correctly rounded sum divided by the count.
#include <cuda_fp16.h>
#include <limits.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <vector>

#include "cp_async.cuh"
#include "f32x2.cuh"
#include "seedq_internal.cuh"
#include "synth.cuh"

namespace seedq {
namespace {

constexpr int kTC = 32;                        // columns per tile
constexpr int kCT = 256;                       // threads per CTA of the column pass
constexpr int kPhases = kCT / 4;               // row phases (4 threads x 8 columns per row)
constexpr int kUnroll = 8;                     // rows per thread per stage
constexpr int kStageRows = kUnroll * kPhases;  // 512
constexpr int kRing = 3;                       // stages in the ring
constexpr int kHS = 257;                       // histogram row stride (bank spread)
constexpr int kGH = 64;                        // Gauss-Hermite nodes
constexpr int kMaxJobs = 4;
constexpr double kEpsDR = 5.9604644775390625e-08;  // 2^-24
constexpr double kDrMin = 1.0e3;
constexpr double kActMin = 1.0e2;

__constant__ float c_gh_xf[kGH];  // Gauss-Hermite nodes
__constant__ float c_gh_wf[kGH];  // weights / sqrt(pi)

// Compensated float32 sum (Kahan): s + (-c) carries the running sum to a few
// units in the last place independently of the number of terms.
struct Kahan {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float y = __fsub_rn(x, c);
    const float t = __fadd_rn(s, y);
    c = __fsub_rn(__fsub_rn(t, s), y);
    s = t;
  }
  __device__ __forceinline__ double value() const { return (double)s - (double)c; }
};

struct Cand {
  double v;
  int32_t t, c;
};

// Partial results of one (slab, tile) work item of the column pass.
struct Part {
  double cs[kTC];
  uint32_t mx[kTC], m0[kTC], cnt[kTC];  // cnt: elements below the slab's threshold
};

struct ColJob {
  const uint16_t *W;     // R x C FP16, row-major
  int32_t R, C;
  int32_t cols;          // 1: column sums wanted
  const float *gw;       // row weights of the column sums (nullptr: all 1)
  double *colsum;        // C
  float *colsum_f;       // C float32 copy, or nullptr
  const float *a;        // C weights of the row sums, or nullptr (no row sums)
  float *rowpart;        // (C / 32) x R
  double *dr;            // C, or nullptr
  int32_t tensor;        // model order, for the candidate list
  Cand *cand;            // dynamic-range candidates (nullptr: none kept)
  uint32_t *ncand;
  int32_t item0;         // first work item of this job in the launch
  int32_t slabs;         // row slabs per tile
  int32_t slab_rows;     // rows per slab (a multiple of 512)
  uint32_t *arrive;      // per tile: slabs finished (0 between launches)
  Part *part;            // per (tile, slab): partial results
};

struct ColArgs {
  ColJob j[kMaxJobs];
  int32_t njobs;
  int32_t items;
};

__device__ __forceinline__ uint4 ld_stream16(const void *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint4 lds128(const uint4 *p) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
  return v;
}

__device__ __forceinline__ double half_val(uint32_t bits) {
  return (double)__half2float(__ushort_as_half((unsigned short)bits));
}

// Median filter.  The dynamic-range statistic reaches 1e3 only when the
// column median is below max / 1e3.  Each row slab takes a provisional
// maximum M0_s from its first 512 rows and a threshold U0_s >= 2.01 K M0_s /
// 1e3 (K = 16), and counts |W| < U0_s while it streams (FP16 compares of FP16
// magnitudes, counted exactly).  With M0 = min_s M0_s, whose threshold U0 is
// the smallest, the counts bound the number of elements below U0.  If the
// column maximum M <= K M0 and the counts sum to at most (R-1)/2, both middle
// order statistics are >= U0, so max / (median + eps) <= 1e3 / 2.01: the
// column cannot qualify.  Every other column gets its exact median.
constexpr float kGrowth = 16.f;
constexpr float kLowFrac = 2.01f * kGrowth / 1000.f;

struct Acc {
  double cs[8];     // column sums (fp64)
  uint64_t cf[4];   // current fp32 chunk, packed pairs
  uint64_t av[4];   // row-sum weights a_c, packed pairs
  uint32_t mx[4];   // packed maxima of |W| bits
  __half2 cnt[4];   // counts of |W| < U0 (small integers, exact in FP16)
  __half2 u0[4];    // thresholds
};

// The thread's rows of one stage (kFull: all 8 valid, else the first nu);
// row weights in wst (shared) unless they are all 1.
template <bool kCols, bool kRows, bool kOnes, bool kFull>
__device__ __forceinline__ void stage_rows(const uint4 *slot, const float *wst, int nu,
                                           float *rowpart, Acc &A) {
  // Full stages: every lane takes part in every shuffle (full mask, no
  // reconvergence); partial stages: only the 4 lanes of the row.
  const unsigned quad = kFull ? 0xffffffffu : (0xFu << (threadIdx.x & 28));
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    if (!kFull && u >= nu) break;
    const uint4 w = lds128(slot + u * kCT);
    const uint32_t wd[4] = {w.x, w.y, w.z, w.w};
    const float gr = (kCols && !kOnes) ? wst[u * kPhases] : 1.f;
    const uint64_t g2 = f2_pack(gr, gr);
    uint64_t rs = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t m = wd[q] & 0x7fff7fffu;  // |w| as FP16 bits
      A.mx[q] = __vmaxu2(A.mx[q], m);
      // Count |w| < U0 in FP16 (exact integers up to 2048 per thread and item).
      A.cnt[q] = __hadd2(A.cnt[q], __hlt2(*reinterpret_cast<const __half2 *>(&m), A.u0[q]));
      if (kCols || kRows) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&wd[q]));
        const uint64_t f2 = f2_pack(f.x, f.y);
        const uint64_t s2 = f2_mul(f2, f2);  // exact: squares of FP16 values
        if (kCols) A.cf[q] = f2_fma(s2, g2, A.cf[q]);
        if (kRows) rs = q ? f2_fma(s2, A.av[q], rs) : f2_mul(s2, A.av[q]);
      }
    }
    if (kRows) {
      const float2 h = f2_unpack(rs);
      float v = h.x + h.y;
      v += __shfl_xor_sync(quad, v, 1);
      v += __shfl_xor_sync(quad, v, 2);
      rowpart[u * kPhases] = v;  // the 4 lanes of the row hold the same sum
    }
  }
}

template <bool kCols, bool kRows>
__device__ __forceinline__ void stage_dispatch(const uint4 *slot, const float *wst, bool ones,
                                               int nu, float *rowpart, Acc &A) {
  // The full-mask path only when every lane of the warp has all 8 rows (row
  // counts that are not multiples of 64 leave the last stage ragged).
  if (__all_sync(0xffffffffu, nu == kUnroll)) {
    if (ones) stage_rows<kCols, kRows, true, true>(slot, wst, nu, rowpart, A);
    else stage_rows<kCols, kRows, false, true>(slot, wst, nu, rowpart, A);
  } else {
    if (ones) stage_rows<kCols, kRows, true, false>(slot, wst, nu, rowpart, A);
    else stage_rows<kCols, kRows, false, false>(slot, wst, nu, rowpart, A);
  }
}

__device__ __forceinline__ void flush_chunk(Acc &A) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 c = f2_unpack(A.cf[q]);
    A.cs[2 * q] += (double)c.x;
    A.cs[2 * q + 1] += (double)c.y;
    A.cf[q] = 0;
  }
}

// Reductions over the 64 row phases of a CTA: the 8 lanes of a warp that
// share a column group combine by an xor tree on lane bits 2..4, then the 8
// warps' results are combined in warp order by the first 32 threads.  Fixed
// order, so the result does not depend on scheduling.
__device__ __forceinline__ uint32_t warp_vmax(uint32_t v) {
  v = __vmaxu2(v, __shfl_xor_sync(0xffffffffu, v, 4));
  v = __vmaxu2(v, __shfl_xor_sync(0xffffffffu, v, 8));
  return __vmaxu2(v, __shfl_xor_sync(0xffffffffu, v, 16));
}
__device__ __forceinline__ uint32_t warp_vadd(uint32_t v) {
  v = __vadd2(v, __shfl_xor_sync(0xffffffffu, v, 4));
  v = __vadd2(v, __shfl_xor_sync(0xffffffffu, v, 8));
  return __vadd2(v, __shfl_xor_sync(0xffffffffu, v, 16));
}
__device__ __forceinline__ double warp_dadd(double v) {
  v += __shfl_xor_sync(0xffffffffu, v, 4);
  v += __shfl_xor_sync(0xffffffffu, v, 8);
  return v + __shfl_xor_sync(0xffffffffu, v, 16);
}

// Packed per-thread values of 8 columns (4 words) reduced to one value per
// column of the tile in out[kTC] (max or sum); buf holds 8 x kTC words.
template <bool kMax>
__device__ __forceinline__ void cta_reduce16(const uint32_t (&v)[4], uint32_t *buf, uint32_t *out) {
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5, lc0 = (t & 3) * 8;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t r = kMax ? warp_vmax(v[q]) : warp_vadd(v[q]);
    if (lane < 4) {
      buf[warp * kTC + lc0 + 2 * q] = r & 0xffffu;
      buf[warp * kTC + lc0 + 2 * q + 1] = r >> 16;
    }
  }
  __syncthreads();
  if (t < kTC) {
    uint32_t a = 0;
    for (int w = 0; w < kCT / 32; ++w) a = kMax ? max(a, buf[w * kTC + t]) : a + buf[w * kTC + t];
    out[t] = a;
  }
  __syncthreads();
}

// Exact medians of the flagged columns of a tile: the bins of the top eight
// bits of |W| holding the order statistics k0 and k1, then the low seven bits
// inside those bins (histograms in hist, kTC x kHS words of global scratch).
// Writes the statistic (0 below the threshold) and the candidates.
__device__ void exact_medians(const ColJob &J, int tile, const int *need, const uint32_t *mxv,
                              uint32_t *hist) {
  __shared__ uint32_t s_b[2][kTC], s_below[2][kTC];
  const int t = threadIdx.x, cg = t & 3, rp = t >> 2, lc0 = cg * 8;
  const int64_t R = J.R, C = J.C;
  const uint16_t *base = J.W + (int64_t)tile * kTC + lc0;
  const uint32_t k0 = (uint32_t)((R - 1) / 2), k1 = (uint32_t)(R / 2);
  for (int i = t; i < kTC * kHS; i += kCT) hist[i] = 0u;
  __syncthreads();
  for (int64_t r = rp; r < R; r += kPhases) {
    const uint4 v4 = ld_stream16(base + r * C);
    const uint32_t wd[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int lc = lc0 + e;
      if (!need[lc]) continue;
      const uint32_t v = ((e & 1) ? wd[e >> 1] >> 16 : wd[e >> 1]) & 0x7fffu;
      atomicAdd(hist + lc * kHS + (v >> 7), 1u);
    }
  }
  __syncthreads();
  if (t < kTC && need[t]) {
    const uint32_t *h = hist + t * kHS;
    uint32_t cum = 0, b0 = 0, b1 = 0, n0 = 0, n1 = 0;
    bool f0 = false, f1 = false;
    for (int b = 0; b < 256; ++b) {
      const uint32_t n = h[b];
      if (!f0 && cum + n > k0) { b0 = b; n0 = cum; f0 = true; }
      if (!f1 && cum + n > k1) { b1 = b; n1 = cum; f1 = true; }
      cum += n;
    }
    s_b[0][t] = b0; s_b[1][t] = b1; s_below[0][t] = n0; s_below[1][t] = n1;
  }
  __syncthreads();
  uint32_t *h2 = hist;  // kTC x 2 x 128
  for (int i = t; i < kTC * 256; i += kCT) h2[i] = 0u;
  __syncthreads();
  for (int64_t r = rp; r < R; r += kPhases) {
    const uint4 v4 = ld_stream16(base + r * C);
    const uint32_t wd[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int lc = lc0 + e;
      if (!need[lc]) continue;
      const uint32_t v = ((e & 1) ? wd[e >> 1] >> 16 : wd[e >> 1]) & 0x7fffu;
      if ((v >> 7) == s_b[0][lc]) atomicAdd(h2 + lc * 256 + (v & 127u), 1u);
      if ((v >> 7) == s_b[1][lc]) atomicAdd(h2 + lc * 256 + 128 + (v & 127u), 1u);
    }
  }
  __syncthreads();
  if (t < kTC && need[t]) {
    uint32_t low[2];
    for (int s = 0; s < 2; ++s) {
      const uint32_t want = (s ? k1 : k0) - s_below[s][t];
      uint32_t cum = 0, l = 0;
      for (; l < 128; ++l) {
        const uint32_t n = h2[t * 256 + s * 128 + l];
        if (cum + n > want) break;
        cum += n;
      }
      low[s] = l;
    }
    const double m1 = half_val((s_b[0][t] << 7) | low[0]);
    const double m2 = half_val((s_b[1][t] << 7) | low[1]);
    const double med = (m1 + m2) * 0.5;
    const double dr = __ddiv_rn(half_val(mxv[t]), __dadd_rn(med, kEpsDR));
    const bool keep = dr >= kDrMin;
    const int64_t col = (int64_t)tile * kTC + t;
    if (J.dr) J.dr[col] = keep ? dr : 0.0;
    if (keep && J.cand) {
      const uint32_t slot = atomicAdd(J.ncand, 1u);
      J.cand[slot] = Cand{dr, J.tensor, (int32_t)col};
    }
  }
  __syncthreads();
}

// A CTA's work: items blockIdx.x, blockIdx.x + gridDim.x, ...; each item a
// row slab of one 32-column tile, streamed in stages of 512 rows.
struct ItemRef {
  int item, job, tile, slab, nst, r_begin, r_end;
};

__device__ __forceinline__ bool item_at(const ColArgs &A, int item, ItemRef &it) {
  if (item >= A.items) return false;
  int ji = 0;
  while (ji + 1 < A.njobs && item >= A.j[ji + 1].item0) ++ji;
  const ColJob &J = A.j[ji];
  // Slab-major: CTAs that run together read the same rows of neighbouring
  // tiles, so each DRAM page they open serves many of them.
  const int local = item - J.item0, tiles = J.C / kTC;
  it.item = item;
  it.job = ji;
  it.slab = local / tiles;
  it.tile = local - it.slab * tiles;
  it.r_begin = it.slab * J.slab_rows;
  it.r_end = min(J.R, it.r_begin + J.slab_rows);
  it.nst = (it.r_end - it.r_begin + kStageRows - 1) / kStageRows;
  return true;
}

// Producer state of the item being issued, in registers: the thread copies
// its own 16-byte piece of each of its rows (and reads back only those); the
// threads of column group 0 also copy the row weights.
struct Feed {
  const uint16_t *src;  // next row's piece
  const float *gsrc;    // next row's weight (nullptr: none copied)
  int64_t step;         // elements between the thread's rows
  int left;             // rows of the item left for this thread
};

__device__ __forceinline__ int rows_of_thread(int r_begin, int r_end, int rp) {
  const int n = r_end - r_begin - rp;
  return n > 0 ? (n + kPhases - 1) / kPhases : 0;
}

__device__ __forceinline__ void feed_start(const ColArgs &A, const ItemRef &it, Feed &F) {
  const ColJob &J = A.j[it.job];
  const int t = threadIdx.x, rp = t >> 2, cg = t & 3;
  const int r = it.r_begin + rp;
  F.src = J.W + (int64_t)r * J.C + it.tile * kTC + cg * 8;
  F.step = (int64_t)kPhases * J.C;
  F.gsrc = (J.cols && J.gw && cg == 0) ? J.gw + r : nullptr;
  F.left = rows_of_thread(it.r_begin, it.r_end, rp);
}

__device__ __forceinline__ void feed_stage(Feed &F, uint4 *slot, float *wslot) {
  const int t = threadIdx.x, rp = t >> 2;
  if (F.left >= kUnroll) {  // the common case: all 8 rows, no per-row branch
    const uint16_t *src = F.src;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      cp_async16(slot + u * kCT + t, src);
      src += F.step;
    }
    F.src = src;
    if (F.gsrc) {
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) cp_async4(wslot + rp + u * kPhases, F.gsrc + u * kPhases);
    }
  } else {
    for (int u = 0; u < F.left; ++u) {
      cp_async16(slot + u * kCT + t, F.src);
      if (F.gsrc) cp_async4(wslot + rp + u * kPhases, F.gsrc + u * kPhases);
      F.src += F.step;
    }
  }
  if (F.gsrc) F.gsrc += kStageRows;
  F.left -= kUnroll;
}

__global__ void __launch_bounds__(kCT, 2) k_colpass(const __grid_constant__ ColArgs A, uint32_t *ghist_all) {
  extern __shared__ uint4 ring[];  // kRing x kUnroll x kCT
  __shared__ float wring[kRing][kStageRows];
  __shared__ uint32_t buf[(kCT / 32) * kTC * 2];
  __shared__ uint32_t s_m0[kTC], s_u0[kTC], s_max[kTC], s_cnt[kTC];
  __shared__ int s_need[kTC];
  __shared__ int s_last, s_any;
  const int t = threadIdx.x, rp = t >> 2, lc0 = (t & 3) * 8;
  uint32_t *ghist = ghist_all + (int64_t)blockIdx.x * kTC * kHS;
  ItemRef pi, ci;
  Feed feed;
  bool p_ok = item_at(A, blockIdx.x, pi);
  int p_stage = 0;
  if (p_ok) feed_start(A, pi, feed);
  auto p_advance = [&]() {
    if (++p_stage == pi.nst) {
      p_stage = 0;
      p_ok = item_at(A, pi.item + gridDim.x, pi);
      if (p_ok) feed_start(A, pi, feed);
    }
  };
  for (int k = 0; k < kRing - 1; ++k) {
    if (p_ok) {
      feed_stage(feed, ring + (size_t)k * kUnroll * kCT, wring[k]);
      p_advance();
    }
    cp_async_commit();
  }
  bool c_ok = item_at(A, blockIdx.x, ci);
  int c_stage = 0, c_left = 0;
  Acc acc;
  for (int s = 0; c_ok; ++s) {
    cp_async_wait<kRing - 2>();
    // Each row's weight is copied and read only by the 4 lanes of that row,
    // all in one warp: a warp barrier makes stage s visible and frees the
    // slots of stage s - 1.
    __syncwarp();
    if (p_ok) {
      const int k = (s + kRing - 1) % kRing;
      feed_stage(feed, ring + (size_t)k * kUnroll * kCT, wring[k]);
      p_advance();
    }
    cp_async_commit();
    const ColJob &J = A.j[ci.job];
    const uint4 *slot = ring + (size_t)(s % kRing) * kUnroll * kCT + t;
    const float *wst = wring[s % kRing] + rp;
    if (c_stage == 0) c_left = rows_of_thread(ci.r_begin, ci.r_end, rp);
    const int nu = min(kUnroll, max(c_left, 0));
    c_left -= kUnroll;
    const bool cols = J.cols != 0, rows = J.a != nullptr, ones = J.gw == nullptr;
    if (c_stage == 0) {
      // Item start: provisional maxima and thresholds from its first stage.
      uint32_t m0[4] = {0u, 0u, 0u, 0u};
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if (u >= nu) break;
        const uint4 w = slot[u * kCT];
        const uint32_t wd[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) m0[q] = __vmaxu2(m0[q], wd[q] & 0x7fff7fffu);
      }
      cta_reduce16<true>(m0, buf, s_m0);
      if (t < kTC)
        s_u0[t] = __half_as_ushort(
            __float2half_ru(kLowFrac * __half2float(__ushort_as_half((unsigned short)s_m0[t]))));
      __syncthreads();
#pragma unroll
      for (int q = 0; q < 8; ++q) acc.cs[q] = 0.0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        acc.cf[q] = 0;
        acc.mx[q] = 0u;
        acc.cnt[q] = __float2half2_rn(0.f);
        const uint32_t u2 = s_u0[lc0 + 2 * q] | (s_u0[lc0 + 2 * q + 1] << 16);
        acc.u0[q] = *reinterpret_cast<const __half2 *>(&u2);
        acc.av[q] = rows ? f2_pack(J.a[ci.tile * kTC + lc0 + 2 * q], J.a[ci.tile * kTC + lc0 + 2 * q + 1])
                         : 0;
      }
    }
    const int row0 = ci.r_begin + c_stage * kStageRows + rp;  // the thread's first row
    float *rowpart = rows ? J.rowpart + (int64_t)ci.tile * J.R + row0 : nullptr;
    if (cols && rows) stage_dispatch<true, true>(slot, wst, ones, nu, rowpart, acc);
    else if (cols) stage_dispatch<true, false>(slot, wst, ones, nu, rowpart, acc);
    else if (rows) stage_dispatch<false, true>(slot, wst, ones, nu, rowpart, acc);
    else stage_dispatch<false, false>(slot, wst, ones, nu, rowpart, acc);
    const bool last = c_stage == ci.nst - 1;
    if (cols && ((c_stage & 1) || last)) flush_chunk(acc);  // at most 16 rows per fp32 chunk

    if (last) {
      // Item end: the item's record, then the tile's combination by the last
      // slab to finish.
      Part &P = J.part[(int64_t)ci.tile * J.slabs + ci.slab];
      if (cols) {
        double *red = reinterpret_cast<double *>(buf);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const double v = warp_dadd(acc.cs[q]);
          if ((t & 31) < 4) red[(t >> 5) * kTC + lc0 + q] = v;
        }
        __syncthreads();
        if (t < kTC) {
          double sum = 0.0;
          for (int w = 0; w < kCT / 32; ++w) sum += red[w * kTC + t];
          P.cs[t] = sum;
        }
        __syncthreads();
      }
      cta_reduce16<true>(acc.mx, buf, s_max);
      uint32_t cnt[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 c = __half22float2(acc.cnt[q]);
        cnt[q] = (uint32_t)c.x | ((uint32_t)c.y << 16);
      }
      cta_reduce16<false>(cnt, buf, s_cnt);
      if (t < kTC) {
        P.mx[t] = s_max[t];
        P.m0[t] = s_m0[t];
        P.cnt[t] = s_cnt[t];
        __threadfence();
      }
      __syncthreads();
      if (t == 0) {
        const uint32_t old = atomicAdd(J.arrive + ci.tile, 1u);
        s_last = old == (uint32_t)(J.slabs - 1);
        s_any = 0;
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        if (t < kTC) {
          const int64_t col = (int64_t)ci.tile * kTC + t;
          const Part *ps = J.part + (int64_t)ci.tile * J.slabs;
          double sum = 0.0;
          uint32_t m = 0, mn = 0xffffu, n = 0;  // n: elements below their slab's threshold
          for (int s2 = 0; s2 < J.slabs; ++s2) {
            if (cols) sum += __ldcg(&ps[s2].cs[t]);
            m = max(m, __ldcg(&ps[s2].mx[t]));
            mn = min(mn, __ldcg(&ps[s2].m0[t]));
            n += __ldcg(&ps[s2].cnt[t]);
          }
          if (cols) {
            J.colsum[col] = sum;
            if (J.colsum_f) J.colsum_f[col] = (float)sum;
          }
          s_max[t] = m;
          const float mf = __half2float(__ushort_as_half((unsigned short)m));
          const float m0f = __half2float(__ushort_as_half((unsigned short)mn));
          const int need = (mf > kGrowth * m0f) || (n > (uint32_t)((J.R - 1) / 2));
          s_need[t] = need;
          if (need) atomicOr(&s_any, 1);
          else if (J.dr) J.dr[col] = 0.0;
          if (t == 0) J.arrive[ci.tile] = 0u;  // every slab has arrived: ready for the next launch
        }
        __syncthreads();
        if (s_any) exact_medians(J, ci.tile, s_need, s_max, ghist);
      }
    }
    if (++c_stage == ci.nst) {
      c_stage = 0;
      c_ok = item_at(A, ci.item + gridDim.x, ci);
    }
  }
  cp_async_wait<0>();
}

// Stream-scale bookkeeping.  The backward proxy grows the residual scale by a
// model-dependent factor per layer (tens for Llama shapes), past the float32
// range after a few dozen layers.  Each finishing step therefore scales the
// new stream scale by 2^-e, e the largest binary exponent of the previous one
// (recorded by the step that produced it), which keeps every value below a
// few hundred.  The branch sums that enter a step were computed from the
// previous scale as stored, so they are scaled by the same power of two; such
// scaling changes no rounding, and rho is stored normalized to unit mean
// within its tensor, so the scales cancel.
struct FinArgs {
  const double *G_old;   // d_model, previous stream scale, or nullptr (head step)
  const int *e_old;      // its largest binary exponent
  const double *gx0, *gx1;
  double *G_new;         // d_model (head step: already holds the head's sums)
  float *gf_new;         // float32 copy: the row weights of the next column pass
  int *e_new;            // largest binary exponent of G_new (atomic max)
  double *rho_raw;       // d_model copy of G_new (rho before normalization), or nullptr
  int32_t d;
  // a_down (mode 0) from the gate / up partial row sums, or a_o (mode 1)
  const float *rp0, *rp1;
  int32_t ntile;         // partial-sum tiles (C / 32)
  int32_t nrows;         // rows of the partial sums
  float *a_out;
  int32_t mode;
  int32_t n_out, n_rep, head_dim;
};

// Blocks [0, nb_g) update the stream scale; the rest take 32 output channels
// of a_down / a_o each (tile sums and quadrature split over 8 thread groups,
// combined in a fixed order).  E[silu(g)^2] is evaluated in float32 (each
// term to a few units in the last place, the sum compensated), below the
// tables' tolerance.
__global__ void k_fin(const __grid_constant__ FinArgs f, int nb_g) {
  if ((int)blockIdx.x < nb_g) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    int e = INT_MIN;
    if (i < f.d) {
      double g = f.G_new[i];
      if (f.G_old) {
        g = f.G_old[i] + f.gx0[i];
        if (f.gx1) g = g + f.gx1[i];
        g = scalbn(g, -*f.e_old);
        f.G_new[i] = g;
      }
      f.gf_new[i] = (float)g;
      if (g > 0.0) e = ilogb(g);
      if (f.rho_raw) f.rho_raw[i] = g;
    }
    e = __reduce_max_sync(0xffffffffu, e);
    if ((threadIdx.x & 31) == 0 && e != INT_MIN) atomicMax(f.e_new, e);
    return;
  }
  if (!f.a_out) return;
  // 32 channels per block: thread (cl, tg) sums the tiles tg, tg + 8, ... of
  // channel cl (coalesced across cl); the 8 partial sums are combined in tg
  // order.  All sums are compensated float32 sums (Kahan), accurate to a few
  // units in the last place whatever their length, on the wide float32 pipe.
  __shared__ float red_v[8][32], red_vc[8][32], red_u[8][32], red_uc[8][32];
  __shared__ float s_sd[32];
  __shared__ double s_u[32];
  const int cl = threadIdx.x & 31, tg = threadIdx.x >> 5;
  const int i = ((int)blockIdx.x - nb_g) * 32 + cl;
  const bool ok = i < f.n_out;
  int row = i;
  if (f.mode == 1 && ok) {
    const int h = i / f.head_dim, o = i - h * f.head_dim;
    row = (h / f.n_rep) * f.head_dim + o;
  }
  Kahan v, u;
  if (ok) {
    for (int t = tg; t < f.ntile; t += 8) {
      v.add(f.rp0[(int64_t)t * f.nrows + row]);
      if (f.mode == 0) u.add(f.rp1[(int64_t)t * f.nrows + row]);
    }
  }
  red_v[tg][cl] = v.s; red_vc[tg][cl] = v.c;
  red_u[tg][cl] = u.s; red_uc[tg][cl] = u.c;
  __syncthreads();
  if (tg == 0) {
    Kahan sv, su;
    for (int k = 0; k < 8; ++k) {
      sv.add(red_v[k][cl]);
      sv.add(-red_vc[k][cl]);
      su.add(red_u[k][cl]);
      su.add(-red_uc[k][cl]);
    }
    const double vv = sv.value(), uu = su.value();
    if (f.mode == 1) {
      if (ok) f.a_out[i] = (float)vv;
    } else {
      s_sd[cl] = sqrtf((float)(2.0 * vv));
      s_u[cl] = uu;
    }
  }
  if (f.mode == 1) return;
  __syncthreads();
  // E[silu(g)^2]: the 64 nodes split over the 8 thread groups, float32.
  const float sd = s_sd[cl];
  Kahan acc;
  for (int k = tg; k < kGH; k += 8) {
    const float g = sd * c_gh_xf[k];
    const float y = g / (1.f + expf(-g));
    acc.add(c_gh_wf[k] * (y * y));
  }
  __syncthreads();
  red_v[tg][cl] = acc.s;
  red_vc[tg][cl] = acc.c;
  __syncthreads();
  if (tg == 0 && ok) {
    Kahan e;
    for (int k = 0; k < 8; ++k) {
      e.add(red_v[k][cl]);
      e.add(-red_vc[k][cl]);
    }
    f.a_out[i] = (float)(e.value() * s_u[cl]);
  }
}

// Value-head weights of the backward proxy: value channel (j, o) collects
// the query heads j * n_rep .. j * n_rep + n_rep - 1 at offset o.
__global__ void k_kvsum(const double *__restrict__ Ga, int kvd, int n_rep, int hd,
                        float *__restrict__ gv) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= kvd) return;
  const int j = i / hd, o = i - j * hd;
  double s = 0.0;
  for (int k = 0; k < n_rep; ++k) s += Ga[(int64_t)(j * n_rep + k) * hd + o];
  gv[i] = (float)s;
}

// Deterministic block sum: each thread adds a strided subset in order, then a
// fixed xor tree inside each warp and the warp sums in warp order.
__device__ double block_sum(const double *__restrict__ v, int n) {
  __shared__ double part[32];
  __shared__ double total;
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += v[i];
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += part[w];
    total = t;
  }
  __syncthreads();
  return total;
}

// rho tables: each vector divided by its mean, float32.  Block 2l is rho_o of
// layer l, block 2l + 1 rho_down.
__global__ void k_norm_rho(const double *__restrict__ raw, int d, float *__restrict__ rho_o,
                           float *__restrict__ rho_down) {
  const double *v = raw + (int64_t)blockIdx.x * d;
  float *out = ((blockIdx.x & 1) ? rho_down : rho_o) + (int64_t)(blockIdx.x >> 1) * d;
  const double mean = block_sum(v, d) / (double)d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) out[i] = (float)(v[i] / mean);
}

// Eq. gamma: a = gamma^2 (exact in float32 for FP16 gamma).
__global__ void k_gain_sq(const uint16_t *__restrict__ g, int n, float *__restrict__ a) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) {
    const float v = __half2float(__ushort_as_half(g[i]));
    a[i] = v * v;
  }
}

struct RatioJob {
  const float *a;
  int32_t C;
  int64_t off;  // first column in model order
};

// Correctly rounded sum of non-negative finite float32 values.  Each value is
// sig * 2^(e - 150) with an integer significand sig < 2^24 and biased exponent
// e (subnormals: e = 1); the significands are summed exactly per exponent in
// 64-bit integers, the 255 sums combined exactly in a 320-bit integer in units
// of 2^-149, and the total rounded once to the nearest double (ties to even).
constexpr int kWide = 5;

__device__ void wide_add_shifted(uint64_t (&w)[kWide], uint64_t v, int sh) {
  const int q = sh >> 6, r = sh & 63;
  uint64_t parts[2] = {v << r, r ? v >> (64 - r) : 0ull};
  uint64_t carry = 0;
  for (int i = q; i < kWide; ++i) {
    const uint64_t add = (i - q < 2 ? parts[i - q] : 0ull);
    const uint64_t s1 = w[i] + add;
    const uint64_t c1 = s1 < add;
    const uint64_t s2 = s1 + carry;
    const uint64_t c2 = s2 < carry;
    w[i] = s2;
    carry = c1 + c2;
    if (i - q >= 1 && !carry) break;
  }
}

__device__ bool wide_bit(const uint64_t (&w)[kWide], int i) {
  return (w[i >> 6] >> (i & 63)) & 1ull;
}

__device__ double wide_round(const uint64_t (&w)[kWide]) {
  int p = -1;
  for (int i = kWide - 1; i >= 0 && p < 0; --i)
    if (w[i]) p = 64 * i + 63 - __clzll((long long)w[i]);
  if (p < 0) return 0.0;
  if (p < 53) return ldexp((double)w[0], -149);
  uint64_t m = 0;
  for (int i = p; i >= p - 52; --i) m = (m << 1) | (uint64_t)wide_bit(w, i);
  const bool guard = wide_bit(w, p - 53);
  bool sticky = false;
  for (int i = p - 54; i >= 0 && !sticky; --i) sticky = wide_bit(w, i);
  if (guard && (sticky || (m & 1ull))) {
    ++m;
    if (m >> 53) {
      m >>= 1;
      ++p;
    }
  }
  return ldexp((double)m, p - 52 - 149);
}

__device__ double exact_sum(const float *__restrict__ v, int n) {
  __shared__ unsigned long long bucket[256];
  __shared__ double total;
  for (int i = threadIdx.x; i < 256; i += blockDim.x) bucket[i] = 0ull;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  for (int base = 0; base < n; base += blockDim.x) {
    const int i = base + threadIdx.x;
    uint32_t e = 0, sig = 0;
    if (i < n) {
      const uint32_t b = __float_as_uint(v[i]);
      e = b >> 23;
      sig = b & 0x7fffffu;
      if (e) sig |= 0x800000u;
      else e = 1;
    }
    const unsigned act = __ballot_sync(0xffffffffu, i < n);
    if (i < n) {
      const unsigned grp = __match_any_sync(act, e);
      const uint32_t sum = __reduce_add_sync(grp, sig);
      if (lane == __ffs(grp) - 1) atomicAdd(bucket + e, (unsigned long long)sum);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    uint64_t w[kWide] = {0, 0, 0, 0, 0};
    for (int e = 1; e < 255; ++e)
      if (bucket[e]) wide_add_shifted(w, bucket[e], e - 1);
    total = wide_round(w);
  }
  __syncthreads();
  return total;
}

// Activation statistic a_j / mean(a); one CTA per tensor.
__global__ void k_act_ratio(const RatioJob *__restrict__ jobs, double *__restrict__ ratio,
                            Cand *__restrict__ cand, uint32_t *__restrict__ ncand) {
  const RatioJob J = jobs[blockIdx.x];
  const double mean = exact_sum(J.a, J.C) / (double)J.C;
  for (int c = threadIdx.x; c < J.C; c += blockDim.x) {
    const double r = (double)J.a[c] / mean;
    if (ratio) ratio[J.off + c] = r;
    if (r >= kActMin) {
      const uint32_t slot = atomicAdd(ncand, 1u);
      cand[slot] = Cand{r, (int32_t)blockIdx.x, c};
    }
  }
}

__global__ void k_synth_fp16(uint64_t key, int64_t first, int64_t n, float scale,
                             uint16_t *__restrict__ out) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t h = splitmix64_at(key, (uint64_t)(first + i));
    const int32_t z = (int32_t)((h & 0xffffu) + ((h >> 16) & 0xffffu) + ((h >> 32) & 0xffffu) +
                                (h >> 48)) - 131070;
    out[i] = __half_as_ushort(__float2half_rn((float)z * scale));
  }
}

// ---------------------------------------------------------------- host side

// Gauss-Hermite rule for the weight exp(-x^2) (Golub & Welsch 1969): the
// nodes are the eigenvalues of the Jacobi matrix of the orthonormal Hermite
// polynomials (zero diagonal, off-diagonal sqrt(k/2)), found one by one by
// bisection on the Sturm count; the weights are the Christoffel numbers
// 1 / sum_{k<n} p_k(x)^2.  Returned weights are divided by sqrt(pi) so that
// sum_i w_i f(x_i) approximates E[f(Z / sqrt 2)], Z ~ N(0, 1).
void gauss_hermite(int n, double *x, double *w) {
  auto below = [n](double v) {
    int cnt = 0;
    double q = 1.0;
    for (int i = 0; i < n; ++i) {
      q = (i == 0) ? -v : -v - 0.5 * i / q;
      if (q == 0.0) q = -1e-300;
      if (q < 0.0) ++cnt;
    }
    return cnt;
  };
  const double bound = 2.0 * sqrt(0.5 * (n - 1)) + 1.0;
  const double pi = 3.14159265358979323846;
  for (int k = 0; k < n; ++k) {
    double lo = -bound, hi = bound;
    for (int it = 0; it < 200; ++it) {
      const double mid = 0.5 * (lo + hi);
      if (mid <= lo || mid >= hi) break;
      if (below(mid) >= k + 1) hi = mid;
      else lo = mid;
    }
    const double xv = 0.5 * (lo + hi);
    double p0 = pow(pi, -0.25), p1 = sqrt(2.0) * xv * p0, s = p0 * p0;
    for (int j = 1; j < n; ++j) {
      s += p1 * p1;
      const double p2 = (sqrt(2.0) * xv * p1 - sqrt((double)j) * p0) / sqrt((double)(j + 1));
      p0 = p1;
      p1 = p2;
    }
    x[k] = xv;
    w[k] = 1.0 / s / sqrt(pi);
  }
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

// Work items of a job for slab height h: one per (slab, tile).
int64_t items_of(int64_t R, int64_t C, int64_t h) { return (C / kTC) * ((R + h - 1) / h); }

// Rows per work item of one launch: among the slab heights (multiples of
// kStageRows, at most 2048 rows per thread and item so the FP16 counts stay
// exact), the one whose assignment of items to CTAs (item i to CTA i mod the
// grid, items job by job and slab-major within a job, as the kernel takes
// them) leaves the smallest busiest CTA, each item counting its rows plus
// kItemRows for its fixed work (first-stage maxima, end reductions, record,
// the ring refill across the item boundary).  kItemRows is set by
// measurement: whole passes over the Llama-2-7B and Llama-3-8B shapes took
// 9.39 / 8.87 ms at 256, 7.13 / 7.69 at 768, 7.09 / 7.49 at 2048 and
// 6.93 / 7.41 at 3072 (the choices do not change from 3072 to 4096), against
// 7.79 / 8.40 with about one item per resident CTA.  Launches of one shape
// recur every layer, so the choice is cached per shape.
constexpr int64_t kItemRows = 3072;

int64_t slab_rows_for(const ColArgs &A, int ctas) {
  std::vector<int64_t> key{(int64_t)ctas};
  int64_t maxR = 0;
  for (int i = 0; i < A.njobs; ++i) {
    key.push_back(A.j[i].R);
    key.push_back(A.j[i].C);
    maxR = std::max<int64_t>(maxR, A.j[i].R);
  }
  static std::mutex mu;
  static std::map<std::vector<int64_t>, int64_t> cache;
  {
    std::lock_guard<std::mutex> lk(mu);
    const auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  const int64_t hmax = std::min<int64_t>((maxR + kStageRows - 1) / kStageRows * kStageRows, 2048 * kPhases);
  std::vector<int64_t> load(ctas);
  int64_t best_h = kStageRows, best = -1;
  int64_t last_slabs = -1;
  for (int64_t h = kStageRows; h <= hmax; h += kStageRows) {
    const int64_t slabs0 = (maxR + h - 1) / h;
    if (slabs0 == last_slabs) continue;  // same split of the tallest job as a smaller h
    last_slabs = slabs0;
    int64_t items = 0;
    for (int i = 0; i < A.njobs; ++i) items += items_of(A.j[i].R, A.j[i].C, h);
    const int64_t G = std::min<int64_t>(items, ctas);
    std::fill(load.begin(), load.end(), 0);
    int64_t i = 0;
    for (int jb = 0; jb < A.njobs; ++jb) {
      const int64_t R = A.j[jb].R, tiles = A.j[jb].C / kTC, sl = (R + h - 1) / h;
      for (int64_t s = 0; s < sl; ++s) {
        const int64_t rows = std::min<int64_t>(h, R - s * h) + kItemRows;
        for (int64_t t = 0; t < tiles; ++t, ++i) load[i % G] += rows;
      }
    }
    const int64_t m = *std::max_element(load.begin(), load.begin() + G);
    if (best < 0 || m < best) {
      best = m;
      best_h = h;
    }
  }
  std::lock_guard<std::mutex> lk(mu);
  cache[key] = best_h;
  return best_h;
}

// Device scratch of the column pass: one record per work item and one arrival
// counter per tile (zero between launches).
struct ColScratch {
  Part *part;
  uint32_t *arrive;
  uint32_t *ghist;  // per CTA: kTC x kHS histogram words of the exact-median path
  int64_t part_cap, arrive_cap;
  int ctas;
};

constexpr size_t kRingBytes = sizeof(uint4) * kRing * kUnroll * kCT;

int resident_ctas() {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return 2 * (sms > 0 ? sms : 1);
}

seedq_status launch_cols(ColArgs &A, const ColScratch &S, cudaStream_t st) {
  const int64_t h = slab_rows_for(A, S.ctas);
  int64_t items = 0, tiles = 0;
  for (int i = 0; i < A.njobs; ++i) {
    ColJob &J = A.j[i];
    J.item0 = (int32_t)items;
    J.slab_rows = (int32_t)h;
    J.slabs = (int32_t)((J.R + h - 1) / h);
    J.part = S.part + items;
    J.arrive = S.arrive + tiles;
    items += items_of(J.R, J.C, h);
    tiles += J.C / kTC;
  }
  if (items > S.part_cap || tiles > S.arrive_cap) return SEEDQ_ERR_INVALID_ARG;
  if (items == 0) return SEEDQ_OK;
  A.items = (int32_t)items;
  // Per call: the attribute belongs to the current device.
  const cudaError_t attr = cudaFuncSetAttribute(
      k_colpass, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kRingBytes);
  if (attr != cudaSuccess) return cuda_fail(attr);
  k_colpass<<<(int)std::min<int64_t>(items, S.ctas), kCT, kRingBytes, st>>>(A, S.ghist);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SEEDQ_OK : cuda_fail(e);
}

ColJob stats_job(const uint16_t *W, int64_t R, int32_t C, double *dr, int32_t tensor, Cand *cand,
                 uint32_t *ncand) {
  ColJob j;
  memset(&j, 0, sizeof j);
  j.W = W;
  j.R = R;
  j.C = C;
  j.dr = dr;
  j.tensor = tensor;
  j.cand = cand;
  j.ncand = ncand;
  return j;
}

// Stream-ordered device scratch, freed on the stream when it goes out of scope.
struct DevBuf {
  cudaStream_t st;
  std::vector<void *> ptrs;
  explicit DevBuf(cudaStream_t s) : st(s) {}
  ~DevBuf() {
    for (void *p : ptrs) cudaFreeAsync(p, st);
  }
  template <class T>
  T *get(size_t n, seedq_status *rc) {
    void *p = nullptr;
    if (*rc != SEEDQ_OK) return nullptr;
    const cudaError_t e = cudaMallocAsync(&p, n * sizeof(T) + 16, st);
    if (e != cudaSuccess) {
      cudaGetLastError();
      *rc = e == cudaErrorMemoryAllocation ? SEEDQ_ERR_NOMEM : cuda_fail(e);
      return nullptr;
    }
    ptrs.push_back(p);
    return (T *)p;
  }
};

// The 64-node rule (nodes, then weights / sqrt(pi)) in float32, computed once
// per process in fp64.
const float *gh_rule() {
  static float table[2 * kGH];
  static const bool done = [] {
    double x[kGH], w[kGH];
    gauss_hermite(kGH, x, w);
    for (int k = 0; k < kGH; ++k) {
      table[k] = (float)x[k];
      table[kGH + k] = (float)w[k];
    }
    return true;
  }();
  (void)done;
  return table;
}

}  // namespace
}  // namespace seedq

using namespace seedq;

extern "C" {

seedq_status seedq_synth_fp16(uint64_t key, int64_t first, int64_t n, int32_t m, int32_t e,
                              uint16_t *out, void *cuda_stream) {
  if (n < 0 || first < 0 || m < 1 || m > 63 || e < 0 || e > 40) return SEEDQ_ERR_INVALID_ARG;
  if (n == 0) return SEEDQ_OK;
  if (!out || !aligned16(out)) return SEEDQ_ERR_INVALID_ARG;
  const float scale = ldexpf((float)m, -e);
  const int64_t want = (n + 255) / 256;
  k_synth_fp16<<<(int)std::min<int64_t>(want, 152 * 16), 256, 0, (cudaStream_t)cuda_stream>>>(
      key, first, n, scale, out);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SEEDQ_OK : cuda_fail(err);
}

seedq_status seedq_column_stats(const uint16_t *W, int64_t R, int64_t C, const float *g,
                                double *dyn_range, double *col_sq, void *cuda_stream) {
  if (!W || !dyn_range || !aligned16(W) || R < 1 || R > (1ll << 31) - 1 || C < kTC ||
      C % kTC != 0 || C > (1 << 20))
    return SEEDQ_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  seedq_status rc = SEEDQ_OK;
  DevBuf B(st);
  ColScratch S;
  S.part_cap = items_of(R, C, kStageRows);
  S.arrive_cap = C / kTC;
  S.part = B.get<Part>((size_t)S.part_cap, &rc);
  S.arrive = B.get<uint32_t>((size_t)S.arrive_cap, &rc);
  S.ctas = resident_ctas();
  S.ghist = B.get<uint32_t>((size_t)S.ctas * kTC * kHS, &rc);
  if (rc != SEEDQ_OK) return rc;
  SEEDQ_CUDA(cudaMemsetAsync(S.arrive, 0, sizeof(uint32_t) * S.arrive_cap, st));
  ColArgs A;
  memset(&A, 0, sizeof A);
  A.njobs = 1;
  A.j[0] = stats_job(W, R, (int32_t)C, dyn_range, 0, nullptr, nullptr);
  if (col_sq) {
    A.j[0].cols = 1;
    A.j[0].gw = g;
    A.j[0].colsum = col_sq;
  }
  return launch_cols(A, S, st);
}

seedq_status seedq_importance(const seedq_llama_model *m, const seedq_importance_out *out,
                              seedq_outlier *outliers, int32_t max_outliers, int32_t *n_outliers,
                              void *cuda_stream) {
  if (!m || !out || !m->layers || !m->lm_head || !m->final_norm) return SEEDQ_ERR_INVALID_ARG;
  if (!out->a_o || !out->a_down || !out->rho_o || !out->rho_down) return SEEDQ_ERR_INVALID_ARG;
  if (max_outliers < 0 || (max_outliers > 0 && (!outliers || !n_outliers)))
    return SEEDQ_ERR_INVALID_ARG;
  const int L = m->n_layers, d = m->d_model, H = m->n_heads, KV = m->n_kv_heads, hd = m->head_dim,
            f = m->d_ff;
  const int64_t V = m->vocab;
  if (L < 1 || L > 4096 || d < kTC || d % kTC || f < kTC || f % kTC || H < 1 || KV < 1 ||
      H % KV || hd < 1 || (int64_t)H * hd > (1 << 20) || ((int64_t)H * hd) % kTC ||
      V < 1 || V > (1ll << 31) - 1 || d > (1 << 20) || f > (1 << 20))
    return SEEDQ_ERR_INVALID_ARG;
  const int qd = H * hd, kvd = KV * hd, n_rep = H / KV;
  for (int l = 0; l < L; ++l) {
    const seedq_llama_layer &y = m->layers[l];
    const void *ps[] = {y.wq, y.wk, y.wv, y.wo, y.wgate, y.wup, y.wdown};
    for (const void *p : ps)
      if (!p || !aligned16(p)) return SEEDQ_ERR_INVALID_ARG;
    if (!y.attn_norm || !y.mlp_norm) return SEEDQ_ERR_INVALID_ARG;
  }
  if (!aligned16(m->lm_head)) return SEEDQ_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;

  // Tensor shapes in model order and their first column in model order.
  const int nt = 7 * L + 1;
  std::vector<int64_t> rows(nt), colsv(nt), off(nt + 1, 0);
  for (int l = 0; l < L; ++l) {
    const int64_t r[7] = {qd, kvd, kvd, d, f, f, d};
    const int64_t c[7] = {d, d, d, qd, d, d, f};
    for (int k = 0; k < 7; ++k) {
      rows[7 * l + k] = r[k];
      colsv[7 * l + k] = c[k];
    }
  }
  rows[7 * L] = V;
  colsv[7 * L] = d;
  for (int t = 0; t < nt; ++t) off[t + 1] = off[t] + colsv[t];
  const int64_t total_cols = off[nt];

  seedq_status rc = SEEDQ_OK;
  DevBuf B(st);
  // Column-pass scratch sized for the largest launch below.
  ColScratch S;
  {
    const int64_t u = kStageRows;
    const int64_t it[5] = {items_of(V, d, u), items_of(d, f, u), 2 * items_of(f, d, u),
                           items_of(d, qd, u) + items_of(qd, d, u) + items_of(kvd, d, u),
                           items_of(kvd, d, u)};
    const int64_t tl[5] = {d / kTC, f / kTC, 2 * (d / kTC), qd / kTC + 2 * (d / kTC), d / kTC};
    S.part_cap = *std::max_element(it, it + 5);
    S.arrive_cap = *std::max_element(tl, tl + 5);
    S.part = B.get<Part>((size_t)S.part_cap, &rc);
    S.arrive = B.get<uint32_t>((size_t)S.arrive_cap, &rc);
    S.ctas = resident_ctas();
    S.ghist = B.get<uint32_t>((size_t)S.ctas * kTC * kHS, &rc);
  }
  double *Gbuf = B.get<double>((size_t)2 * d, &rc), *gxa = B.get<double>(d, &rc),
         *gxb = B.get<double>(d, &rc);
  double *Gh = B.get<double>(f, &rc), *Ga = B.get<double>(qd, &rc);
  float *gfs = B.get<float>(d, &rc), *ghf = B.get<float>(f, &rc), *gaf = B.get<float>(qd, &rc);
  float *gvf = n_rep > 1 ? B.get<float>(kvd, &rc) : gaf;
  double *rraw = B.get<double>((size_t)2 * L * d, &rc);  // rho_o of layer l at 2l, rho_down at 2l+1
  int *gexp = B.get<int>((size_t)2 * L + 1, &rc);
  float *rpa = B.get<float>((size_t)(d / kTC) * std::max(f, kvd), &rc);
  float *rpb = B.get<float>((size_t)(d / kTC) * f, &rc);
  float *again = B.get<float>((size_t)(2 * L + 1) * d, &rc);
  Cand *cand = B.get<Cand>((size_t)2 * total_cols, &rc);
  uint32_t *ncand = B.get<uint32_t>(2, &rc);
  RatioJob *djobs = B.get<RatioJob>(nt, &rc);
  if (rc != SEEDQ_OK) return rc;
  Cand *cand_dr = cand, *cand_act = cand + total_cols;
  SEEDQ_CUDA(cudaMemsetAsync(S.arrive, 0, sizeof(uint32_t) * S.arrive_cap, st));
  SEEDQ_CUDA(cudaMemcpyToSymbolAsync(c_gh_xf, gh_rule(), sizeof(float) * kGH, 0,
                                     cudaMemcpyHostToDevice, st));
  SEEDQ_CUDA(cudaMemcpyToSymbolAsync(c_gh_wf, gh_rule() + kGH, sizeof(float) * kGH, 0,
                                     cudaMemcpyHostToDevice, st));
  SEEDQ_CUDA(cudaMemsetAsync(ncand, 0, 2 * sizeof(uint32_t), st));
  SEEDQ_CUDA(cudaMemsetAsync(gexp, 0x80, sizeof(int) * (2 * L + 1), st));  // below any exponent
  const int gb = (d + 255) / 256;
  for (int l = 0; l < L; ++l) {
    k_gain_sq<<<gb, 256, 0, st>>>(m->layers[l].attn_norm, d, again + (size_t)(2 * l) * d);
    k_gain_sq<<<gb, 256, 0, st>>>(m->layers[l].mlp_norm, d, again + (size_t)(2 * l + 1) * d);
  }
  float *a_final = again + (size_t)2 * L * d;
  k_gain_sq<<<gb, 256, 0, st>>>(m->final_norm, d, a_final);
  SEEDQ_CUDA(cudaGetLastError());
  auto drp = [&](int t) { return out->dyn_range ? out->dyn_range + off[t] : nullptr; };
  auto job = [&](int t, const uint16_t *W) {
    return stats_job(W, rows[t], (int32_t)colsv[t], drp(t), t, cand_dr, ncand);
  };
  // The stream scale alternates between two buffers; step s (0 = after the
  // head, then two per layer) has largest exponent gexp[s]; gfs always holds
  // the float32 copy of the current one.
  int step = 0;
  auto Gcur = [&]() { return Gbuf + (size_t)(step & 1) * d; };
  auto Gnext = [&]() { return Gbuf + (size_t)((step + 1) & 1) * d; };

  // The head: an isotropic gradient at the logits gives the stream scale.
  {
    ColArgs A;
    memset(&A, 0, sizeof A);
    A.njobs = 1;
    A.j[0] = job(7 * L, m->lm_head);
    A.j[0].cols = 1;
    A.j[0].colsum = Gcur();
    if ((rc = launch_cols(A, S, st)) != SEEDQ_OK) return rc;
    FinArgs F;
    memset(&F, 0, sizeof F);
    F.G_new = Gcur();
    F.gf_new = gfs;
    F.e_new = gexp;
    F.rho_raw = rraw + (size_t)(2 * (L - 1) + 1) * d;
    F.d = d;
    k_fin<<<gb, 256, 0, st>>>(F, gb);
    SEEDQ_CUDA(cudaGetLastError());
  }
  for (int l = L - 1; l >= 0; --l) {
    const seedq_llama_layer &y = m->layers[l];
    const int t0 = 7 * l;
    const float *a_attn = again + (size_t)(2 * l) * d, *a_mlp = again + (size_t)(2 * l + 1) * d;
    ColArgs A;
    // Down projection: its rows read the stream scale; columns give Gh.
    memset(&A, 0, sizeof A);
    A.njobs = 1;
    A.j[0] = job(t0 + 6, y.wdown);
    A.j[0].cols = 1;
    A.j[0].gw = gfs;
    A.j[0].colsum = Gh;
    A.j[0].colsum_f = ghf;
    if ((rc = launch_cols(A, S, st)) != SEEDQ_OK) return rc;
    // Gate and up: back-map of Gh, and the row sums of Eq. prop.
    memset(&A, 0, sizeof A);
    A.njobs = 2;
    A.j[0] = job(t0 + 4, y.wgate);
    A.j[1] = job(t0 + 5, y.wup);
    for (int i = 0; i < 2; ++i) {
      A.j[i].cols = 1;
      A.j[i].gw = ghf;
      A.j[i].colsum = i ? gxb : gxa;
      A.j[i].a = a_mlp;
      A.j[i].rowpart = i ? rpb : rpa;
    }
    if ((rc = launch_cols(A, S, st)) != SEEDQ_OK) return rc;
    {
      FinArgs F;
      memset(&F, 0, sizeof F);
      F.G_old = Gcur(); F.e_old = gexp + step; F.gx0 = gxa; F.gx1 = gxb;
      F.G_new = Gnext(); F.gf_new = gfs; F.e_new = gexp + step + 1;
      F.rho_raw = rraw + (size_t)(2 * l) * d; F.d = d;
      F.rp0 = rpa; F.rp1 = rpb; F.ntile = d / kTC; F.nrows = f;
      F.a_out = out->a_down + (size_t)l * f; F.mode = 0; F.n_out = f;
      k_fin<<<gb + (f + 31) / 32, 256, 0, st>>>(F, gb);
      SEEDQ_CUDA(cudaGetLastError());
      ++step;
    }
    // Output projection (stream scale in, attention scale out) with the
    // statistics of q and k.
    memset(&A, 0, sizeof A);
    A.njobs = 3;
    A.j[0] = job(t0 + 3, y.wo);
    A.j[0].cols = 1;
    A.j[0].gw = gfs;
    A.j[0].colsum = Ga;
    A.j[0].colsum_f = gaf;
    A.j[1] = job(t0 + 0, y.wq);
    A.j[2] = job(t0 + 1, y.wk);
    if ((rc = launch_cols(A, S, st)) != SEEDQ_OK) return rc;
    if (n_rep > 1) {
      k_kvsum<<<(kvd + 255) / 256, 256, 0, st>>>(Ga, kvd, n_rep, hd, gvf);
      SEEDQ_CUDA(cudaGetLastError());
    }
    // Value projection: rows weighted by the query heads of each value head,
    // and the row sums of a^(o).
    memset(&A, 0, sizeof A);
    A.njobs = 1;
    A.j[0] = job(t0 + 2, y.wv);
    A.j[0].cols = 1;
    A.j[0].gw = gvf;
    A.j[0].colsum = gxa;
    A.j[0].a = a_attn;
    A.j[0].rowpart = rpa;
    if ((rc = launch_cols(A, S, st)) != SEEDQ_OK) return rc;
    {
      FinArgs F;
      memset(&F, 0, sizeof F);
      F.G_old = Gcur(); F.e_old = gexp + step; F.gx0 = gxa;
      F.G_new = Gnext(); F.gf_new = gfs; F.e_new = gexp + step + 1;
      F.rho_raw = l > 0 ? rraw + (size_t)(2 * (l - 1) + 1) * d : nullptr; F.d = d;
      F.rp0 = rpa; F.ntile = d / kTC; F.nrows = kvd;
      F.a_out = out->a_o + (size_t)l * qd; F.mode = 1; F.n_out = qd;
      F.n_rep = n_rep; F.head_dim = hd;
      k_fin<<<gb + (qd + 31) / 32, 256, 0, st>>>(F, gb);
      SEEDQ_CUDA(cudaGetLastError());
      ++step;
    }
  }
  // Stored rho: unit mean within each tensor.
  k_norm_rho<<<2 * L, 256, 0, st>>>(rraw, d, out->rho_o, out->rho_down);
  SEEDQ_CUDA(cudaGetLastError());

  // Activation statistic of every tensor.
  std::vector<RatioJob> hj(nt);
  for (int l = 0; l < L; ++l) {
    const float *a_attn = again + (size_t)(2 * l) * d, *a_mlp = again + (size_t)(2 * l + 1) * d;
    const float *as[7] = {a_attn, a_attn, a_attn, out->a_o + (size_t)l * qd, a_mlp, a_mlp,
                          out->a_down + (size_t)l * f};
    for (int k = 0; k < 7; ++k) hj[7 * l + k] = RatioJob{as[k], (int32_t)colsv[7 * l + k], off[7 * l + k]};
  }
  hj[7 * L] = RatioJob{a_final, d, off[7 * L]};
  SEEDQ_CUDA(cudaMemcpyAsync(djobs, hj.data(), sizeof(RatioJob) * nt, cudaMemcpyHostToDevice, st));
  k_act_ratio<<<nt, 256, 0, st>>>(djobs, out->act_ratio, cand_act, ncand + 1);
  SEEDQ_CUDA(cudaGetLastError());

  // App. A.6 selection on the host over the (few) candidates.
  uint32_t nc[2] = {0, 0};
  SEEDQ_CUDA(cudaMemcpyAsync(nc, ncand, sizeof nc, cudaMemcpyDeviceToHost, st));
  SEEDQ_CUDA(cudaStreamSynchronize(st));
  std::vector<Cand> lists[2];
  for (int r = 0; r < 2; ++r) {
    lists[r].resize(nc[r]);
    if (nc[r])
      SEEDQ_CUDA(cudaMemcpy(lists[r].data(), r ? cand_act : cand_dr, sizeof(Cand) * nc[r],
                            cudaMemcpyDeviceToHost));
    std::sort(lists[r].begin(), lists[r].end(), [](const Cand &x, const Cand &y) {
      if (x.v != y.v) return x.v > y.v;
      if (x.t != y.t) return x.t < y.t;
      return x.c < y.c;
    });
    if (lists[r].size() > 32) lists[r].resize(32);
  }
  struct Ranked {
    int pos;
    int32_t t, c;
  };
  std::vector<Ranked> merged;
  for (int r = 0; r < 2; ++r)
    for (size_t p = 0; p < lists[r].size(); ++p) {
      const Cand &x = lists[r][p];
      bool found = false;
      for (Ranked &y : merged)
        if (y.t == x.t && y.c == x.c) {
          y.pos = std::min(y.pos, (int)p);
          found = true;
        }
      if (!found) merged.push_back(Ranked{(int)p, x.t, x.c});
    }
  std::sort(merged.begin(), merged.end(), [](const Ranked &x, const Ranked &y) {
    if (x.pos != y.pos) return x.pos < y.pos;
    if (x.t != y.t) return x.t < y.t;
    return x.c < y.c;
  });
  if (n_outliers) {
    const int n = std::min<int>((int)merged.size(), max_outliers);
    for (int i = 0; i < n; ++i) outliers[i] = seedq_outlier{merged[i].t, merged[i].c};
    *n_outliers = n;
  }
  return SEEDQ_OK;
}

}  // extern "C"
