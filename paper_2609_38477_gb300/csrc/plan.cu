// Decoder plan of Alg. 2 (imp, floor, ladder, tie pass, row offsets), LFSR jump
// tables, layer lifetime and the synthetic stream generator.
#include <cuda_fp16.h>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <vector>

#include "seedq_internal.cuh"
#include "synth.cuh"

namespace seedq {

static thread_local char g_last_cuda_error[256] = "";

seedq_status cuda_fail(cudaError_t e) {
  snprintf(g_last_cuda_error, sizeof g_last_cuda_error, "%s: %s", cudaGetErrorName(e),
           cudaGetErrorString(e));
  return SEEDQ_ERR_CUDA;
}

// Feedback taps of the width-S LFSR of the stream format: o_{t+S} = XOR over
// set bits i of o_{t+i}.  Each is a primitive polynomial x^S + sum x^i with the
// smallest possible largest tap below S (so one machine word yields the most
// new sequence bits per step), then the fewest taps, then the smallest mask.
static const uint32_t kTaps[17] = {0, 0, 0, 0, 0, 0, 0, 0,
                                   0x1d,  // S=8:  x^8+x^4+x^3+x^2+1
                                   0x11,  // S=9:  x^9+x^4+1
                                   0x09,  // S=10: x^10+x^3+1
                                   0x05,  // S=11: x^11+x^2+1
                                   0x53,  // S=12: x^12+x^6+x^4+x+1
                                   0x1b,  // S=13: x^13+x^4+x^3+x+1
                                   0x2b,  // S=14: x^14+x^5+x^3+x+1
                                   0x03,  // S=15: x^15+x+1
                                   0x2d}; // S=16: x^16+x^5+x^3+x^2+1

// ------------------------------------------------------------ plan kernels

// Stable ranking of n keys in O(n log n): every chunk of kRankChunk keys is
// sorted by (key, index) in shared memory (bitonic network), then each key's
// rank is the number of entries below it in every sorted chunk (a binary
// search per chunk), and out[rank] = its index.  The order is ascending keys
// (kDesc: descending), ties by ascending index:
//   perm:    columns by ascending a (Sec. 3.3: channels sorted by a before
//            blocking), perm[rank] = column;
//   rowperm: the fused kernel's row order, rows by decreasing rho, so rows
//            with equal or nearby rung breakpoints (monotone in imp = abar *
//            rho) share a warp; with no row factor the natural order is kept.
// One launch serves several jobs (blocks located by binary search over their
// first-block numbers).
constexpr int kRankChunk = 1024;

template <typename K>
struct RankJob {
  const K *key;
  int32_t *out;     // n: out[rank] = index
  K *skey;          // scratch: n keys in sorted chunks
  int32_t *sidx;    // scratch: their indices
  int32_t n;
  int32_t sblk0;    // first block of this job in the sort launch (one per chunk)
  int32_t rblk0;    // first block of this job in the rank launch (256 keys each)
};

template <typename K, bool kDesc>
__device__ __forceinline__ bool rank_less(K ka, int32_t ia, K kb, int32_t ib) {
  // Padding entries (index -1) sort after every key.
  if (ia < 0) return false;
  if (ib < 0) return true;
  if (ka != kb) return kDesc ? ka > kb : ka < kb;
  return ia < ib;
}

template <typename K>
__device__ __forceinline__ int rank_job(const RankJob<K> *jobs, int nj, int b, bool sort_launch) {
  int lo = 0, hi = nj - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if ((sort_launch ? jobs[mid].sblk0 : jobs[mid].rblk0) <= b) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

template <typename K, bool kDesc>
__global__ void __launch_bounds__(kRankChunk / 2) k_chunk_sort(const RankJob<K> *__restrict__ jobs, int nj) {
  __shared__ K sk[kRankChunk];
  __shared__ int32_t si[kRankChunk];
  const RankJob<K> &J = jobs[rank_job(jobs, nj, blockIdx.x, true)];
  const int base = (blockIdx.x - J.sblk0) * kRankChunk;
  for (int t = threadIdx.x; t < kRankChunk; t += blockDim.x) {
    const int i = base + t;
    sk[t] = i < J.n ? J.key[i] : K(0);
    si[t] = i < J.n ? i : -1;
  }
  __syncthreads();
  for (int k = 2; k <= kRankChunk; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      const int t = threadIdx.x;
      const int i = ((t & ~(j - 1)) << 1) | (t & (j - 1)), l = i + j;
      const bool up = (i & k) == 0;
      const bool sw = up ? rank_less<K, kDesc>(sk[l], si[l], sk[i], si[i])
                         : rank_less<K, kDesc>(sk[i], si[i], sk[l], si[l]);
      if (sw) {
        const K tk = sk[i];
        sk[i] = sk[l];
        sk[l] = tk;
        const int32_t ti = si[i];
        si[i] = si[l];
        si[l] = ti;
      }
      __syncthreads();
    }
  }
  for (int t = threadIdx.x; t < kRankChunk && base + t < J.n; t += blockDim.x) {
    J.skey[base + t] = sk[t];
    J.sidx[base + t] = si[t];
  }
}

template <typename K, bool kDesc>
__global__ void __launch_bounds__(256) k_chunk_rank(const RankJob<K> *__restrict__ jobs, int nj) {
  const RankJob<K> &J = jobs[rank_job(jobs, nj, blockIdx.x, false)];
  const int i = (blockIdx.x - J.rblk0) * 256 + threadIdx.x;
  if (i >= J.n) return;
  const K ki = J.key[i];
  int rank = 0;
  for (int c0 = 0; c0 < J.n; c0 += kRankChunk) {
    int lo = 0, hi = min(kRankChunk, J.n - c0);
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (rank_less<K, kDesc>(J.skey[c0 + mid], J.sidx[c0 + mid], ki, i)) lo = mid + 1;
      else hi = mid;
    }
    rank += lo;
  }
  J.out[rank] = i;
}

// Launches the two kernels over nj jobs whose descriptors (with block numbers
// filled in by this function) go to d_jobs.
template <typename K, bool kDesc>
static cudaError_t launch_rank(RankJob<K> *h_jobs, int nj, RankJob<K> *d_jobs, cudaStream_t st) {
  int sb = 0, rbk = 0;
  for (int t = 0; t < nj; ++t) {
    h_jobs[t].sblk0 = sb;
    h_jobs[t].rblk0 = rbk;
    sb += (h_jobs[t].n + kRankChunk - 1) / kRankChunk;
    rbk += (h_jobs[t].n + 255) / 256;
  }
  cudaError_t e = cudaMemcpyAsync(d_jobs, h_jobs, sizeof(RankJob<K>) * nj, cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess || sb == 0) return e;
  k_chunk_sort<K, kDesc><<<sb, kRankChunk / 2, 0, st>>>(d_jobs, nj);
  k_chunk_rank<K, kDesc><<<rbk, 256, 0, st>>>(d_jobs, nj);
  return cudaGetLastError();
}

__global__ void k_iota(int64_t n, int32_t *__restrict__ out) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = (int32_t)i;
}

// The fused kernel's per-row record, in its row order: row r = rowperm[i] at
// position i, with its bit offset and breakpoints in two 16-byte words, so a
// warp fetches its 32 rows' plan data with two contiguous loads per lane.
__global__ void k_rowrec(const int32_t *__restrict__ rowperm, const uint64_t *__restrict__ row_off,
                         const int32_t *__restrict__ brk, int J, int64_t R, uint4 *__restrict__ rec) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < R;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = rowperm[i];
    const uint64_t off = row_off[r];
    const uint32_t row_bits = (uint32_t)(row_off[r + 1] - off);
    static_assert(kMaxJ == 9, "the record holds eight breakpoints");
    uint32_t b[kMaxJ - 1];
#pragma unroll
    for (int j = 0; j < kMaxJ - 1; ++j)
      b[j] = j < J - 1 ? (uint32_t)(uint16_t)brk[r * (J - 1) + j] : 0x7fffu;
    rec[2 * i] = make_uint4((uint32_t)off, (uint32_t)(off >> 32), b[0] | (b[1] << 16), b[2] | (b[3] << 16));
    rec[2 * i + 1] = make_uint4(b[4] | (b[5] << 16), b[6] | (b[7] << 16), row_bits, 0u);
  }
}

__global__ void k_invperm(const int32_t *__restrict__ perm, int C, int32_t *__restrict__ inv) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < C) inv[perm[i]] = i;
}

// Block means of the permuted a, summed in channel order, and their unit-mean
// normalization summed in ascending block order (Eq. imp; App. A.7 fixed order).
// One thread block per tensor.
__device__ __forceinline__ void abar_block(const float *__restrict__ a, const int32_t *__restrict__ perm,
                                           int nb, double *__restrict__ abar) {
  __shared__ double mean;
  for (int c = threadIdx.x; c < nb; c += blockDim.x) {
    double s = 0.0;
    for (int i = 0; i < 8; ++i) s = __dadd_rn(s, (double)a[perm[8 * c + i]]);
    abar[c] = __ddiv_rn(s, 8.0);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int c = 0; c < nb; ++c) s = __dadd_rn(s, abar[c]);
    mean = __ddiv_rn(s, (double)nb);
  }
  __syncthreads();
  for (int c = threadIdx.x; c < nb; c += blockDim.x) abar[c] = __ddiv_rn(abar[c], mean);
}

__global__ void k_abar(const float *__restrict__ a, const int32_t *__restrict__ perm,
                       int nb, double *__restrict__ abar) {
  abar_block(a, perm, nb, abar);
}

// Row factor normalized to unit mean, summed in ascending row order.
__device__ __forceinline__ void rho_block(const float *__restrict__ rho_in, int64_t R,
                                          double *__restrict__ rho) {
  __shared__ double mean;
  if (threadIdx.x == 0) {
    double s = 0.0;
    if (rho_in)
      for (int64_t r = 0; r < R; ++r) s = __dadd_rn(s, (double)rho_in[r]);
    mean = __ddiv_rn(s, (double)R);
  }
  __syncthreads();
  for (int64_t r = threadIdx.x; r < R; r += blockDim.x)
    rho[r] = rho_in ? __ddiv_rn((double)rho_in[r], mean) : 1.0;
}

__global__ void k_rho(const float *__restrict__ rho_in, int64_t R, double *__restrict__ rho) {
  rho_block(rho_in, R, rho);
}

// The same three steps for many tensors at once (the allocator's factors).
struct FacJob {
  const float *a;       // C
  const float *rho_in;  // R, or nullptr
  int32_t *perm;        // C
  double *abar;         // C / 8
  double *rho;          // R
  int64_t R;
  int32_t C;
};

__global__ void k_factors_multi(const FacJob *__restrict__ jobs) {
  const FacJob &J = jobs[blockIdx.x];
  abar_block(J.a, J.perm, J.C / 8, J.abar);
  __syncthreads();
  rho_block(J.rho_in, J.R, J.rho);
}

struct SchedArgs {
  int J;
  int j_tie;
  double q;
  double theta[kMaxJ];
};

// Floored importance of block c of a row with factor rr: max(abar_c * rho_r, q).
__device__ __forceinline__ double imp_at(const double *abar, double rr, double q, int c) {
  const double v = __dmul_rn(abar[c], rr);
  return (v < q) ? q : v;
}

// First block of the row whose importance is >= thr (> thr when strict);
// importance is non-decreasing along a row because channels are sorted.
__device__ int first_block(const double *abar, double rr, double q, int nb, double thr,
                           bool strict) {
  int lo = 0, hi = nb;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    const double v = imp_at(abar, rr, q, mid);
    const bool pass = strict ? (v > thr) : (v >= thr);
    if (pass) hi = mid;
    else lo = mid + 1;
  }
  return lo;
}

// Eq. ladder as breakpoints: brk[r][j] = first block with theta_j <= imp, i.e.
// rung >= j+1; tcnt[r] = blocks of the row tied at theta[j_tie].
__global__ void k_rows(const double *__restrict__ abar, const double *__restrict__ rho,
                       int nb, int64_t R, SchedArgs s, int32_t *__restrict__ brk,
                       int32_t *__restrict__ tcnt) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  const double rr = rho[r];
  for (int j = 0; j < s.J - 1; ++j)
    brk[r * (s.J - 1) + j] = first_block(abar, rr, s.q, nb, s.theta[j], false);
  int t = 0;
  if (s.j_tie >= 0) {
    const int hi = first_block(abar, rr, s.q, nb, s.theta[s.j_tie], true);
    t = hi - brk[r * (s.J - 1) + s.j_tie];
  }
  tcnt[r] = t;
}

// Block-wide exclusive scan of per-thread totals (1024 threads).
__device__ uint64_t block_exclusive_scan(uint64_t v, uint64_t *sh, uint64_t *total) {
  const int t = threadIdx.x;
  sh[t] = v;
  __syncthreads();
  for (int d = 1; d < blockDim.x; d <<= 1) {
    const uint64_t add = (t >= d) ? sh[t - d] : 0;
    __syncthreads();
    sh[t] += add;
    __syncthreads();
  }
  const uint64_t incl = sh[t];
  if (total) *total = sh[blockDim.x - 1];
  __syncthreads();
  return incl - v;
}

// Tie pass of Alg. 2 (the first T tied blocks in row-major order take the lower
// rung) applied to the breakpoints, then per-row bit counts and their exclusive
// scan into row offsets.  One CTA of 1024 threads, rows in contiguous chunks.
// Block bits of each rung, passed by value in the kernel's parameters.
struct RungBits {
  int32_t L[kMaxJ];
};

__global__ void k_scan(int64_t R, int J, int nb, int j_tie, int64_t T, const RungBits Lrung,
                       int32_t *__restrict__ brk, const int32_t *__restrict__ tcnt,
                       uint64_t *__restrict__ row_off, uint64_t *__restrict__ summary) {
  __shared__ uint64_t sh[1024];
  __shared__ int L[kMaxJ];
  if (threadIdx.x < J) L[threadIdx.x] = Lrung.L[threadIdx.x];
  const int64_t per = (R + blockDim.x - 1) / blockDim.x;
  const int64_t r0 = min((int64_t)threadIdx.x * per, R), r1 = min(r0 + per, R);
  uint64_t tied_total = 0;
  if (j_tie >= 0) {
    uint64_t local = 0;
    for (int64_t r = r0; r < r1; ++r) local += (uint64_t)tcnt[r];
    uint64_t prefix = block_exclusive_scan(local, sh, &tied_total);
    for (int64_t r = r0; r < r1; ++r) {
      const int64_t left = T - (int64_t)prefix;
      const int64_t d = left <= 0 ? 0 : (left < tcnt[r] ? left : tcnt[r]);
      brk[r * (J - 1) + j_tie] += (int32_t)d;
      prefix += (uint64_t)tcnt[r];
    }
  }
  __syncthreads();
  uint64_t local = 0;
  for (int64_t r = r0; r < r1; ++r) {
    uint64_t b = (uint64_t)L[0] * (uint64_t)nb;
    for (int j = 0; j < J - 1; ++j)
      b += (uint64_t)(L[j + 1] - L[j]) * (uint64_t)(nb - brk[r * (J - 1) + j]);
    local += b;
  }
  uint64_t total = 0;
  uint64_t off = block_exclusive_scan(local, sh, &total);
  for (int64_t r = r0; r < r1; ++r) {
    row_off[r] = off;
    uint64_t b = (uint64_t)L[0] * (uint64_t)nb;
    for (int j = 0; j < J - 1; ++j)
      b += (uint64_t)(L[j + 1] - L[j]) * (uint64_t)(nb - brk[r * (J - 1) + j]);
    off += b;
  }
  if (threadIdx.x == 0) {
    row_off[R] = total;
    summary[0] = tied_total;
    summary[1] = total;
  }
}

// GF(2) jump tables: tab[v] = first 64 sequence bits from seed v, tab[256+v]
// from seed v << 8; by linearity the prefix of any seed is the XOR of the two.
__global__ void k_tables(const int32_t *__restrict__ slot_S, uint64_t *__restrict__ tables,
                         uint32_t t0, uint32_t t1, uint32_t t2, uint32_t t3, uint32_t t4,
                         uint32_t t5, uint32_t t6, uint32_t t7, uint32_t t8) {
  const uint32_t taps_arr[9] = {t0, t1, t2, t3, t4, t5, t6, t7, t8};
  const int slot = blockIdx.x;
  const int S = slot_S[slot];
  const uint32_t taps = taps_arr[S - 8];
  const int v = threadIdx.x;  // 0..511
  tables[(size_t)slot * 512 + v] = jump_table_entry(S, taps, v);
}

// Synthetic payload of the workload recipe, one thread per block.

__global__ void k_synth(const __grid_constant__ LayerArgs p, const int32_t *__restrict__ S_of, const int32_t *__restrict__ K_of,
                        uint64_t key, uint32_t *__restrict__ out) {
  const int64_t total = p.R * (int64_t)p.nb;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < total;
       b += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = b / p.nb;
    const int c = (int)(b - r * p.nb);
    int32_t bk[kMaxJ];
    for (int j = 0; j < p.J - 1; ++j) bk[j] = p.brk[r * (p.J - 1) + j];
    const int g = rung_of(bk, p.J, c);
    const int S = S_of[g], K = K_of[g];
    const uint64_t off = p.row_off[r] + bits_before(bk, p.J, p.L, p.nb, c);
    const uint64_t h = splitmix64_at(key, (uint64_t)b);
    const uint32_t seed = 1u + (uint32_t)(h >> 32) % ((1u << S) - 1u);
    const int E = -8 + (int)(((h >> 24) & 255u) % 6u);
    uint64_t v = (uint64_t)seed | ((uint64_t)(E & 15) << S);
    for (int j = 0; j < K; ++j) {
      const int t = (int)((h >> (4 * j)) & 15u) - 8;
      v |= (uint64_t)(t & 15) << (S + 4 + 4 * j);
    }
    const uint64_t wi = off >> 5;
    const int sh = (int)(off & 31);
    atomicOr(out + wi, (uint32_t)(v << sh));
    const uint64_t rest = (sh == 0) ? (v >> 32) : (v >> (32 - sh));
    if (rest) atomicOr(out + wi + 1, (uint32_t)rest);
    const uint64_t rest2 = (sh == 0) ? 0 : (v >> (64 - sh));
    if (sh && rest2) atomicOr(out + wi + 2, (uint32_t)rest2);
  }
}

static void free_layer(seedq_layer *L) {
  if (!L) return;
  cudaFree(L->d_perm);
  cudaFree(L->d_invperm);
  cudaFree(L->d_abar);
  cudaFree(L->d_rho);
  cudaFree(L->d_rho_in);
  cudaFree(L->d_a_in);
  cudaFree(L->d_brk);
  cudaFree(L->d_tcnt);
  cudaFree(L->d_row_off);
  cudaFree(L->d_tables);
  cudaFree(L->d_flags);
  cudaFree(L->d_summary);
  cudaFree(L->d_rowperm);
  cudaFree(L->d_rowrec);
  cudaFree(L->d_counters);
  cudaFree(L->d_slots);
  cudaFree(L->d_xperm);
  free(L->h_gp);
  free(L->h_gk);
  free(L->h_repbk);

  free(L);
}


// Host-side work profile of the tensor for the fused kernel's partition.
// Units are (row group, block) pairs in row-group-major order.  The kernel
// walks a row group's blocks in stages of a few columns; where all 32 rows of
// the group sit at one rung it makes one pass per block, and from the first
// column where they differ to the end of the stage it makes, for each rung
// present, as many passes as the row with the most blocks at that rung in the
// stage.  The profile counts those passes (stages aligned at block 0) and the
// sum of k over them, per row group; the first row's breakpoints are kept to
// place a cost target inside a group.
static seedq_status build_costs(seedq_layer *L, cudaStream_t st) {
  const int64_t R = L->args.R;
  const int J = L->args.J, Jm1 = J > 1 ? J - 1 : 1, nb = L->args.nb;
  const int64_t G = (R + 31) / 32;
  int32_t *rowperm = (int32_t *)malloc(sizeof(int32_t) * R);
  int32_t *brk = (int32_t *)malloc(sizeof(int32_t) * R * Jm1);
  L->h_gp = (double *)malloc(sizeof(double) * (G + 1));
  L->h_gk = (double *)malloc(sizeof(double) * (G + 1));
  L->h_repbk = (int32_t *)malloc(sizeof(int32_t) * G * Jm1);
  const int nst = (nb + kCostStage - 1) / kCostStage;
  uint8_t *mixed = (uint8_t *)malloc(nst);
  seedq_status rc = SEEDQ_OK;
  if (!rowperm || !brk || !L->h_gp || !L->h_gk || !L->h_repbk || !mixed) rc = SEEDQ_ERR_NOMEM;
  cudaError_t e = cudaSuccess;
  if (rc == SEEDQ_OK) e = cudaMemcpyAsync(rowperm, L->d_rowperm, sizeof(int32_t) * R, cudaMemcpyDeviceToHost, st);
  if (rc == SEEDQ_OK && e == cudaSuccess && J > 1)
    e = cudaMemcpyAsync(brk, L->d_brk, sizeof(int32_t) * R * Jm1, cudaMemcpyDeviceToHost, st);
  if (rc == SEEDQ_OK && e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) rc = cuda_fail(e);
  if (rc == SEEDQ_OK) {
    L->h_gp[0] = 0.0;
    L->h_gk[0] = 0.0;
    const int32_t *rowb[32];
    for (int64_t g = 0; g < G; ++g) {
      int nr = 0;
      for (int i = 0; i < 32 && g * 32 + i < R; ++i) rowb[nr++] = brk + (int64_t)rowperm[g * 32 + i] * Jm1;
      const int32_t *b0 = rowb[0];
      int32_t *rb = L->h_repbk + g * Jm1;
      // The first row's profile.
      double P = nb, K = 0.0;
      int lo = 0;
      for (int j = 0; j < J; ++j) {
        const int hi = (j < J - 1) ? b0[j] : nb;
        if (j < J - 1) rb[j] = b0[j];
        K += (double)L->k[j] * (hi - lo);
        lo = hi;
      }
      // Stages where the rows' breakpoints differ: replace the first row's
      // passes there by the per-rung maxima over the rows.
      bool any = false;
      for (int s = 0; s < nst; ++s) mixed[s] = 0;
      for (int j = 0; j < J - 1; ++j) {
        int mn = b0[j], mx = b0[j];
        for (int i = 1; i < nr; ++i) {
          mn = rowb[i][j] < mn ? rowb[i][j] : mn;
          mx = rowb[i][j] > mx ? rowb[i][j] : mx;
        }
        if (mn < mx) {
          any = true;
          const int s0 = mn / kCostStage, s1 = (mx - 1) / kCostStage;
          for (int s = s0; s <= s1 && s < nst; ++s) mixed[s] = 1;
        }
      }
      if (any) {
        for (int s = 0; s < nst; ++s) {
          if (!mixed[s]) continue;
          const int cs = s * kCostStage, ce = (cs + kCostStage < nb) ? cs + kCostStage : nb;
          for (int j = 0; j < J; ++j) {
            int mxc = 0, c0 = 0;
            for (int i = 0; i < nr; ++i) {
              const int a = (j > 0) ? rowb[i][j - 1] : 0, z = (j < J - 1) ? rowb[i][j] : nb;
              const int ra = a > cs ? a : cs, rz = z < ce ? z : ce;
              const int cnt = rz > ra ? rz - ra : 0;
              if (i == 0) c0 = cnt;
              mxc = cnt > mxc ? cnt : mxc;
            }
            P += mxc - c0;
            K += (double)L->k[j] * (mxc - c0);
          }
        }
      }
      L->h_gp[g + 1] = L->h_gp[g] + P;
      L->h_gk[g + 1] = L->h_gk[g] + K;
    }
  }
  free(mixed);
  free(rowperm);
  free(brk);
  return rc;
}

}  // namespace seedq

using namespace seedq;

extern "C" {

const char *seedq_status_string(seedq_status s) {
  switch (s) {
    case SEEDQ_OK: return "ok";
    case SEEDQ_ERR_INVALID_ARG: return "invalid argument";
    case SEEDQ_ERR_STREAM: return "stream length or buffer size does not match the plan";
    case SEEDQ_ERR_SCHEDULE: return "inconsistent schedule tables";
    case SEEDQ_ERR_CUDA: return "CUDA error";
    case SEEDQ_ERR_NOMEM: return "out of memory";
    case SEEDQ_ERR_UNSUPPORTED: return "unsupported rung or shape";
    case SEEDQ_ERR_IO: return "container file could not be opened, read or written";
    case SEEDQ_ERR_FORMAT: return "container file is malformed, truncated or corrupted";
  }
  return "unknown status";
}

const char *seedq_last_cuda_error_string(void) { return g_last_cuda_error; }

uint32_t seedq_lfsr_taps(int32_t S) { return (S >= 8 && S <= 16) ? kTaps[S] : 0u; }

uint64_t seedq_stream_bytes_required(uint64_t bits) { return stream_bytes_required(bits); }

seedq_status seedq_layer_prepare(const seedq_layer_desc *d, const seedq_schedule *s,
                                 void *cuda_stream, seedq_layer **out) {
  if (!d || !s || !out) return SEEDQ_ERR_INVALID_ARG;
  *out = nullptr;
  if (d->rows < 1 || d->rows > (1ll << 24) || d->cols < 8 || (d->cols % 8) != 0 || !d->a)
    return SEEDQ_ERR_INVALID_ARG;
  if (d->cols > kMaxCols) return SEEDQ_ERR_UNSUPPORTED;
  if (d->n_outliers < 0 || d->n_outliers > kMaxOutliers) return SEEDQ_ERR_INVALID_ARG;
  if (d->n_outliers > 0 && (!d->outlier_cols || !d->outlier_vals)) return SEEDQ_ERR_INVALID_ARG;
  if (d->tie_count < 0) return SEEDQ_ERR_SCHEDULE;
  const int mb = d->max_batch == 0 ? kMaxBatch : d->max_batch;
  if (mb < 1 || mb > kMaxBatch) return SEEDQ_ERR_INVALID_ARG;
  if (s->J < 1 || s->J > kMaxJ || !s->rungs || (s->J > 1 && !s->theta)) return SEEDQ_ERR_SCHEDULE;
  for (int j = 0; j < s->J; ++j) {
    if (!rung_supported(s->rungs[j].S, s->rungs[j].k)) return SEEDQ_ERR_UNSUPPORTED;
    if (j > 0 && s->rungs[j].S + 4 * s->rungs[j].k <= s->rungs[j - 1].S + 4 * s->rungs[j - 1].k)
      return SEEDQ_ERR_SCHEDULE;
  }
  for (int j = 0; j + 1 < s->J; ++j) {
    if (!isfinite(s->theta[j])) return SEEDQ_ERR_SCHEDULE;
    if (j > 0 && !(s->theta[j] > s->theta[j - 1])) return SEEDQ_ERR_SCHEDULE;
  }
  if (s->j_tie < -1 || s->j_tie >= s->J - 1 || (s->J == 1 && s->j_tie != -1)) return SEEDQ_ERR_SCHEDULE;
  if (!isfinite(s->q)) return SEEDQ_ERR_SCHEDULE;
  double asum = 0.0;
  for (int64_t c = 0; c < d->cols; ++c) {
    if (!isfinite(d->a[c]) || d->a[c] < 0.f) return SEEDQ_ERR_INVALID_ARG;
    asum += d->a[c];
  }
  if (!(asum > 0.0)) return SEEDQ_ERR_INVALID_ARG;
  if (d->rho)
    for (int64_t r = 0; r < d->rows; ++r)
      if (!isfinite(d->rho[r]) || !(d->rho[r] > 0.f)) return SEEDQ_ERR_INVALID_ARG;
  for (int o = 0; o < d->n_outliers; ++o) {
    if (d->outlier_cols[o] < 0 || d->outlier_cols[o] >= d->cols) return SEEDQ_ERR_INVALID_ARG;
    for (int p = 0; p < o; ++p)
      if (d->outlier_cols[p] == d->outlier_cols[o]) return SEEDQ_ERR_INVALID_ARG;
  }

  seedq_layer *L = (seedq_layer *)calloc(1, sizeof(seedq_layer));
  if (!L) return SEEDQ_ERR_NOMEM;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const int64_t R = d->rows, C = d->cols;
  const int nb = (int)(C / 8), J = s->J;
  L->args.R = R;
  L->args.C = C;
  L->args.nb = nb;
  L->args.J = J;
  L->j_tie = s->j_tie;
  L->q = s->q;
  L->tie_count = d->tie_count;
  L->max_batch = mb;
  cudaGetDevice(&L->device);
  // One jump-table slot per supported seed width (8, 10, ..., 16); the tables
  // depend only on S, so every layer's table set is the same.
  const int nslots = kTableSlots;
  for (int t = 0; t < nslots; ++t) L->slot_S[t] = 8 + 2 * t;
  for (int j = 0; j < J; ++j) {
    L->S[j] = s->rungs[j].S;
    L->k[j] = s->rungs[j].k;
    L->args.L[j] = L->S[j] + 4 * L->k[j] + 4;
    L->args.code[j] = rung_code(L->S[j], L->k[j]);
    L->args.slot[j] = (L->S[j] - 8) / 2;
    if (j + 1 < J) L->theta[j] = s->theta[j];
  }
  for (int j = 0; j < kMaxJ - 1; ++j) L->args.dL[j] = j + 1 < J ? L->args.L[j + 1] - L->args.L[j] : 0;
  L->args.nslots = nslots;
  L->args.n_out = d->n_outliers;
  for (int o = 0; o < d->n_outliers; ++o) L->args.out_cols[o] = d->outlier_cols[o];
  L->args.out_vals = d->outlier_vals;

  const int Jm1 = J > 1 ? J - 1 : 1;
  seedq_status rc = SEEDQ_OK;
#define ALLOC(ptr, bytes)                                              \
  do {                                                                 \
    cudaError_t e_ = cudaMalloc((void **)&(ptr), (bytes));             \
    if (e_ != cudaSuccess) {                                           \
      cudaGetLastError();                                              \
      free_layer(L);                                                   \
      return e_ == cudaErrorMemoryAllocation ? SEEDQ_ERR_NOMEM : cuda_fail(e_); \
    }                                                                  \
  } while (0)
  ALLOC(L->d_perm, sizeof(int32_t) * C);
  ALLOC(L->d_invperm, sizeof(int32_t) * C);
  ALLOC(L->d_abar, sizeof(double) * nb);
  ALLOC(L->d_rho, sizeof(double) * R);
  ALLOC(L->d_a_in, sizeof(float) * C);
  if (d->rho) ALLOC(L->d_rho_in, sizeof(float) * R);
  ALLOC(L->d_brk, sizeof(int32_t) * R * Jm1);
  ALLOC(L->d_tcnt, sizeof(int32_t) * R);
  ALLOC(L->d_row_off, sizeof(uint64_t) * (R + 1));
  ALLOC(L->d_tables, sizeof(uint64_t) * 512 * nslots);
  ALLOC(L->d_flags, sizeof(uint32_t));
  ALLOC(L->d_summary, sizeof(uint64_t) * 2);
  {
    int32_t *dS = nullptr;
    ALLOC(dS, sizeof(int32_t) * kMaxJ);
    cudaError_t e = cudaMemcpyAsync(dS, L->slot_S, sizeof(int32_t) * kMaxJ, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) {
      k_tables<<<nslots, 512, 0, st>>>(dS, L->d_tables, kTaps[8], kTaps[9], kTaps[10], kTaps[11],
                                       kTaps[12], kTaps[13], kTaps[14], kTaps[15], kTaps[16]);
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    cudaFree(dS);
    if (e != cudaSuccess) { free_layer(L); return cuda_fail(e); }
  }
  {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    L->max_ctas = sms > 0 ? sms : 1;
  }
  const int64_t ngroups = (R + 31) / 32;
  ALLOC(L->d_rowperm, sizeof(int32_t) * R);
  ALLOC(L->d_rowrec, sizeof(uint4) * 2 * R);
  ALLOC(L->d_counters, sizeof(int32_t) * ngroups);
  ALLOC(L->d_slots, sizeof(float) * L->max_ctas * 2 * 32 * kMaxBatch);
  // Weight-major activations, padded to the kernel's batch template.
  const int mbt = mb <= 1 ? 1 : mb <= 2 ? 2 : mb <= 4 ? 4 : mb <= 8 ? 8 : 16;
  ALLOC(L->d_xperm, sizeof(float) * C * mbt);

#undef ALLOC
  L->args.perm = L->d_perm;
  L->args.rowperm = L->d_rowperm;
  L->args.rowrec = L->d_rowrec;
  L->args.counters = L->d_counters;
  L->args.slots = L->d_slots;
  L->args.xperm = L->d_xperm;
  L->args.invperm = L->d_invperm;
  L->args.brk = L->d_brk;
  L->args.row_off = L->d_row_off;
  L->args.tables = L->d_tables;
  L->args.flags = L->d_flags;

  L->args.stream = nullptr;
  L->args.stream_words = 0;

  RungBits rb;
  for (int j = 0; j < kMaxJ; ++j) rb.L[j] = L->args.L[j];
  bool rho_uniform = true;
  if (d->rho)
    for (int64_t r = 1; r < R; ++r) rho_uniform &= (d->rho[r] == d->rho[0]);
  const bool rank_rows = !rho_uniform && R <= 65536;
  // Scratch of the stable rankings (columns by a, rows by rho), freed below.
  uint8_t *scr = nullptr;
  const size_t scr_cols = (size_t)C * 8, scr_rows = rank_rows ? (size_t)R * 16 : 0;
  const size_t scr_jobs = sizeof(RankJob<float>) + sizeof(RankJob<double>);
  cudaError_t e = cudaMalloc((void **)&scr, scr_cols + scr_rows + scr_jobs);
  if (e != cudaSuccess) {
    free_layer(L);
    return cuda_fail(e);
  }
  if (e == cudaSuccess) e = cudaMemsetAsync(L->d_flags, 0, sizeof(uint32_t), st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(L->d_a_in, d->a, sizeof(float) * C, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && d->rho)
    e = cudaMemcpyAsync(L->d_rho_in, d->rho, sizeof(float) * R, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) {
    RankJob<float> jc{L->d_a_in, L->d_perm, reinterpret_cast<float *>(scr),
                      reinterpret_cast<int32_t *>(scr + (size_t)C * 4), (int32_t)C, 0, 0};
    e = launch_rank<float, false>(&jc, 1, reinterpret_cast<RankJob<float> *>(scr + scr_cols + scr_rows), st);
    k_invperm<<<(int)((C + 255) / 256), 256, 0, st>>>(L->d_perm, (int)C, L->d_invperm);
    k_abar<<<1, 1024, 0, st>>>(L->d_a_in, L->d_perm, nb, L->d_abar);
    k_rho<<<1, 1024, 0, st>>>(L->d_rho_in, R, L->d_rho);
    SchedArgs sa;
    sa.J = J;
    sa.j_tie = s->j_tie;
    sa.q = s->q;
    for (int j = 0; j < kMaxJ; ++j) sa.theta[j] = (j + 1 < J) ? s->theta[j] : 0.0;
    if (J > 1) {
      k_rows<<<(int)((R + 255) / 256), 256, 0, st>>>(L->d_abar, L->d_rho, nb, R, sa, L->d_brk,
                                                     L->d_tcnt);
    } else {
      e = cudaMemsetAsync(L->d_tcnt, 0, sizeof(int32_t) * R, st);
    }
    k_scan<<<1, 1024, 0, st>>>(R, J, nb, J > 1 ? s->j_tie : -1, d->tie_count, rb, L->d_brk,
                               L->d_tcnt, L->d_row_off, L->d_summary);
    if (!rank_rows) {
      k_iota<<<(int)((R + 255) / 256 < 4096 ? (R + 255) / 256 : 4096), 256, 0, st>>>(R, L->d_rowperm);
    } else if (e == cudaSuccess) {
      RankJob<double> jr{L->d_rho, L->d_rowperm, reinterpret_cast<double *>(scr + scr_cols),
                         reinterpret_cast<int32_t *>(scr + scr_cols + (size_t)R * 8), (int32_t)R, 0, 0};
      e = launch_rank<double, true>(
          &jr, 1, reinterpret_cast<RankJob<double> *>(scr + scr_cols + scr_rows + sizeof(RankJob<float>)), st);
    }
    k_rowrec<<<(int)((R + 255) / 256 < 4096 ? (R + 255) / 256 : 4096), 256, 0, st>>>(
        L->d_rowperm, L->d_row_off, L->d_brk, J, R, L->d_rowrec);
    if (e == cudaSuccess) e = cudaMemsetAsync(L->d_counters, 0, sizeof(int32_t) * ngroups, st);
    if (e == cudaSuccess) e = cudaGetLastError();
  }
  uint64_t summary[2] = {0, 0};
  if (e == cudaSuccess) e = cudaMemcpyAsync(summary, L->d_summary, sizeof summary, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e == cudaSuccess) e = cudaFree(scr);
  else cudaFree(scr);
  if (e != cudaSuccess) {
    free_layer(L);
    return cuda_fail(e);
  }
  if (s->j_tie >= 0 && (uint64_t)d->tie_count > summary[0]) rc = SEEDQ_ERR_SCHEDULE;
  if (s->j_tie < 0 && d->tie_count != 0) rc = SEEDQ_ERR_SCHEDULE;
  if (rc != SEEDQ_OK) {
    free_layer(L);
    return rc;
  }
  L->total_bits = summary[1];
  {
    seedq_status prc = build_costs(L, st);
    if (prc != SEEDQ_OK) {
      free_layer(L);
      return prc;
    }
  }
  // The plan's fp32 copies of a and rho are no longer needed.
  cudaFree(L->d_a_in);
  L->d_a_in = nullptr;
  cudaFree(L->d_rho_in);
  L->d_rho_in = nullptr;
  *out = L;
  return SEEDQ_OK;
}

seedq_status seedq_layer_stream_bits(const seedq_layer *L, uint64_t *bits) {
  if (!L || !bits) return SEEDQ_ERR_INVALID_ARG;
  *bits = L->total_bits;
  return SEEDQ_OK;
}

seedq_status seedq_layer_bind_stream(seedq_layer *L, const void *stream, uint64_t bits,
                                     uint64_t bytes) {
  if (!L || !stream) return SEEDQ_ERR_INVALID_ARG;
  if (((uintptr_t)stream & 15u) != 0) return SEEDQ_ERR_INVALID_ARG;
  if (bits != L->total_bits || bytes < stream_bytes_required(bits)) return SEEDQ_ERR_STREAM;
  L->stream = stream;
  L->stream_bytes = bytes;
  L->args.stream = (const uint32_t *)stream;
  L->args.stream_words = bytes / 4;
  return SEEDQ_OK;
}

seedq_status seedq_layer_limit_stream_bytes(seedq_layer *L, uint64_t bytes) {
  if (!L) return SEEDQ_ERR_INVALID_ARG;
  if (!L->args.stream) return SEEDQ_ERR_STREAM;
  if (bytes > L->stream_bytes) return SEEDQ_ERR_INVALID_ARG;
  L->stream_bytes = bytes;
  L->args.stream_words = bytes / 4;
  return SEEDQ_OK;
}

seedq_status seedq_layer_release(seedq_layer *L) {
  if (!L) return SEEDQ_OK;
  cudaError_t e = cudaDeviceSynchronize();
  free_layer(L);
  return e == cudaSuccess ? SEEDQ_OK : cuda_fail(e);
}

seedq_status seedq_layer_rung_map(const seedq_layer *L, int64_t row0, int64_t nrows,
                                  uint8_t *rungs_host) {
  if (!L || !rungs_host || row0 < 0 || nrows < 0 || row0 + nrows > L->args.R)
    return SEEDQ_ERR_INVALID_ARG;
  const int J = L->args.J, nb = L->args.nb, Jm1 = J > 1 ? J - 1 : 1;
  int32_t *bk = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nrows * Jm1 + 1));
  if (!bk) return SEEDQ_ERR_NOMEM;
  if (nrows) {
    cudaError_t e = cudaMemcpy(bk, L->d_brk + row0 * Jm1, sizeof(int32_t) * nrows * Jm1,
                               cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) { free(bk); return cuda_fail(e); }
  }
  for (int64_t i = 0; i < nrows; ++i)
    for (int c = 0; c < nb; ++c) {
      int j = 0;
      for (int t = 0; t < J - 1; ++t) j += (bk[i * Jm1 + t] <= c) ? 1 : 0;
      rungs_host[i * nb + c] = (uint8_t)j;
    }
  free(bk);
  return SEEDQ_OK;
}

seedq_status seedq_layer_perm(const seedq_layer *L, int32_t *perm_host) {
  if (!L || !perm_host) return SEEDQ_ERR_INVALID_ARG;
  SEEDQ_CUDA(cudaMemcpy(perm_host, L->d_perm, sizeof(int32_t) * L->args.C, cudaMemcpyDeviceToHost));
  return SEEDQ_OK;
}

seedq_status seedq_layer_row_offsets(const seedq_layer *L, uint64_t *offs) {
  if (!L || !offs) return SEEDQ_ERR_INVALID_ARG;
  SEEDQ_CUDA(cudaMemcpy(offs, L->d_row_off, sizeof(uint64_t) * (L->args.R + 1), cudaMemcpyDeviceToHost));
  return SEEDQ_OK;
}

seedq_status seedq_last_device_error(const seedq_layer *L, uint32_t *flags) {
  if (!L || !flags) return SEEDQ_ERR_INVALID_ARG;
  SEEDQ_CUDA(cudaMemcpy(flags, L->d_flags, sizeof(uint32_t), cudaMemcpyDeviceToHost));
  return SEEDQ_OK;
}

seedq_status seedq_synth_stream(const seedq_layer *L, uint64_t key, void *stream,
                                uint64_t stream_bytes, void *cuda_stream) {
  if (!L || !stream || ((uintptr_t)stream & 15u)) return SEEDQ_ERR_INVALID_ARG;
  if (stream_bytes < stream_bytes_required(L->total_bits)) return SEEDQ_ERR_STREAM;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  int32_t *dSK = nullptr;
  SEEDQ_CUDA(cudaMalloc((void **)&dSK, sizeof(int32_t) * 2 * kMaxJ));
  int32_t hSK[2 * kMaxJ];
  for (int j = 0; j < kMaxJ; ++j) {
    hSK[j] = L->S[j];
    hSK[kMaxJ + j] = L->k[j];
  }
  cudaError_t e = cudaMemcpyAsync(dSK, hSK, sizeof hSK, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(stream, 0, stream_bytes, st);
  if (e == cudaSuccess) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    k_synth<<<sms * 8, 256, 0, st>>>(L->args, dSK, dSK + kMaxJ, key, (uint32_t *)stream);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(dSK);
  return e == cudaSuccess ? SEEDQ_OK : cuda_fail(e);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free row pass.  Some callers cannot call cudaMalloc at the moment
// they need a plan: code running inside a fixed memory budget reserved up
// front, allocator-less embedded runtimes, or code that must not touch the
// CUDA allocator while other work is in flight.  For them the per-row part of
// the plan (ladder breakpoints, tie pass, row offsets) can run with its
// temporary per-row tie counts kept in this file-scope device array instead of
// layer-owned memory.  Every GPU that loads the library holds the array until
// the process exits.  All calls share it, so calls that overlap on the GPU race.
namespace seedq {

constexpr int64_t kStaticPlanMaxRows = 1 << 17;

struct StaticPlanScratch {
  int32_t tcnt[kStaticPlanMaxRows];
};

static __device__ __align__(256) StaticPlanScratch g_static_plan_scratch;

// Device address of the array on the current device (in host code the symbol
// is only a host-side stand-in).  Looked up on every call: the first lookup on
// a device loads the module there, later ones are cheap, and an address is
// never reused from a context that has since been destroyed.
static StaticPlanScratch *static_scratch_ptr(seedq_status *st) {
  void *p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_static_plan_scratch);
  if (e != cudaSuccess) {
    *st = cuda_fail(e);
    return nullptr;
  }
  *st = SEEDQ_OK;
  return (StaticPlanScratch *)p;
}

}  // namespace seedq

extern "C" seedq_status seedq_row_plan_static(const double *abar, const double *rho, int64_t rows,
                                              int32_t nb, const seedq_schedule *s,
                                              int64_t tie_count, int32_t *brk, uint64_t *row_off,
                                              uint64_t *summary, void *cuda_stream) {
  if (!abar || !rho || !s || !row_off || !summary || rows < 1 || nb < 1) return SEEDQ_ERR_INVALID_ARG;
  if (rows > kStaticPlanMaxRows) return SEEDQ_ERR_UNSUPPORTED;
  if (nb > kMaxCols / 8) return SEEDQ_ERR_UNSUPPORTED;
  if (s->J < 1 || s->J > kMaxJ || !s->rungs || (s->J > 1 && (!s->theta || !brk)))
    return SEEDQ_ERR_SCHEDULE;
  for (int j = 0; j < s->J; ++j) {
    if (!rung_supported(s->rungs[j].S, s->rungs[j].k)) return SEEDQ_ERR_UNSUPPORTED;
    if (j > 0 && s->rungs[j].S + 4 * s->rungs[j].k <= s->rungs[j - 1].S + 4 * s->rungs[j - 1].k)
      return SEEDQ_ERR_SCHEDULE;
  }
  for (int j = 0; j + 1 < s->J; ++j) {
    if (!isfinite(s->theta[j])) return SEEDQ_ERR_SCHEDULE;
    if (j > 0 && !(s->theta[j] > s->theta[j - 1])) return SEEDQ_ERR_SCHEDULE;
  }
  if (s->j_tie < -1 || s->j_tie >= s->J - 1 || !isfinite(s->q) || tie_count < 0) return SEEDQ_ERR_SCHEDULE;
  if (s->j_tie < 0 && tie_count != 0) return SEEDQ_ERR_SCHEDULE;
  seedq_status st = SEEDQ_OK;
  StaticPlanScratch *scr = static_scratch_ptr(&st);
  if (!scr) return st;
  cudaStream_t cs = (cudaStream_t)cuda_stream;
  RungBits rb;
  for (int j = 0; j < kMaxJ; ++j) rb.L[j] = j < s->J ? s->rungs[j].S + 4 * s->rungs[j].k + 4 : 0;
  SchedArgs sa;
  sa.J = s->J;
  sa.j_tie = s->j_tie;
  sa.q = s->q;
  for (int j = 0; j < kMaxJ; ++j) sa.theta[j] = (j + 1 < s->J) ? s->theta[j] : 0.0;
  // k_rows writes every row's tie count before k_scan reads it, so the shared
  // array needs no clearing; with a single rung there are no ties to count.
  if (s->J > 1)
    k_rows<<<(int)((rows + 255) / 256), 256, 0, cs>>>(abar, rho, nb, rows, sa, brk, scr->tcnt);
  k_scan<<<1, 1024, 0, cs>>>(rows, s->J, nb, s->J > 1 ? s->j_tie : -1, tie_count, rb, brk,
                             scr->tcnt, row_off, summary);
  SEEDQ_CUDA(cudaGetLastError());
  return SEEDQ_OK;
}

// ------------------------------------------------------------ allocator
// Alg. 1 over a set of tensors: every count is an integer summed with atomic
// adds and every importance the same fp64 product as the plan's, so the
// bisections take the same steps on any device and agree with a sequential
// evaluation.
namespace seedq {
namespace {

struct AllocTensor {
  const double *abar;  // nb unit-mean block means (ascending)
  const double *rho;   // rows unit-mean row factors
  int64_t R;           // rows of the tensor
  int64_t row0;        // first evaluated row in the launch's row space
  int32_t nrows;       // evaluated rows (1 when rho is 1 on every row)
  int32_t nb;
};

enum AllocMode { kCountLE = 0, kBits = 1, kVmin = 2, kTied = 3 };

struct AllocArgs {
  const AllocTensor *t;
  int32_t nt;
  int64_t rows;        // evaluated rows over all tensors
  int32_t mode, J;
  int32_t L[kMaxJ];
  double q, v;
  double th[kMaxJ];
  unsigned long long *total;      // kCountLE / kBits / kTied: one counter
  unsigned long long *per_tensor; // kBits / kTied: nt counters
  unsigned long long *vmin;       // kVmin: J - 1 bit patterns
};

__global__ void k_alloc_eval(const __grid_constant__ AllocArgs a) {
  const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  unsigned long long val = 0;
  int ti = -1;
  if (g < a.rows) {
    int lo = 0, hi = a.nt - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (a.t[mid].row0 <= g) lo = mid;
      else hi = mid - 1;
    }
    ti = lo;
    const AllocTensor &T = a.t[ti];
    const double rr = T.rho[g - T.row0];
    const unsigned long long mult = T.nrows == 1 ? (unsigned long long)T.R : 1ull;
    if (a.mode == kCountLE) {
      val = (unsigned long long)first_block(T.abar, rr, -INFINITY, T.nb, a.v, true) * mult;
    } else if (a.mode == kBits) {
      unsigned long long rb = (unsigned long long)a.L[0] * (unsigned long long)T.nb;
      for (int j = 0; j < a.J - 1; ++j) {
        const int n_ge = T.nb - first_block(T.abar, rr, a.q, T.nb, a.th[j], false);
        rb += (unsigned long long)(a.L[j + 1] - a.L[j]) * (unsigned long long)n_ge;
      }
      val = rb * mult;
    } else if (a.mode == kTied) {
      val = (unsigned long long)(first_block(T.abar, rr, a.q, T.nb, a.v, true) -
                                 first_block(T.abar, rr, a.q, T.nb, a.v, false)) * mult;
    } else {
      for (int j = 0; j < a.J - 1; ++j) {
        const int c = first_block(T.abar, rr, a.q, T.nb, a.th[j], false);
        if (c < T.nb) atomicMin(a.vmin + j, (unsigned long long)__double_as_longlong(imp_at(T.abar, rr, a.q, c)));
      }
    }
  }
  if (a.mode == kVmin) return;
  if (val && a.per_tensor) atomicAdd(a.per_tensor + ti, val);
  for (int o = 16; o > 0; o >>= 1) val += __shfl_xor_sync(0xffffffffu, val, o);
  if ((threadIdx.x & 31) == 0 && val) atomicAdd(a.total, val);
}

double from_bits(int64_t p) {
  double d;
  memcpy(&d, &p, sizeof d);
  return d;
}

int64_t to_bits(double d) {
  int64_t p;
  memcpy(&p, &d, sizeof p);
  return p;
}

struct Allocator {
  AllocArgs base;
  cudaStream_t st;
  unsigned long long *dev;  // 1 + nt + kMaxJ counters
  int nt;
  seedq_status err = SEEDQ_OK;

  // One evaluation: returns the total; per-tensor counts into pt when given.
  uint64_t run(int mode, double q, double v, const double *th, uint64_t *pt = nullptr,
               double *vmin = nullptr) {
    if (err != SEEDQ_OK) return 0;
    AllocArgs a = base;
    a.mode = mode;
    a.q = q;
    a.v = v;
    for (int j = 0; j < kMaxJ; ++j) a.th[j] = (th && j + 1 < a.J) ? th[j] : 0.0;
    a.total = dev;
    a.per_tensor = pt ? dev + 1 : nullptr;
    a.vmin = dev + 1 + nt;
    std::vector<unsigned long long> init(1 + nt + kMaxJ, 0ull);
    for (int j = 0; j < kMaxJ; ++j) init[1 + nt + j] = (unsigned long long)to_bits(INFINITY);
    cudaError_t e = cudaMemcpyAsync(dev, init.data(), sizeof(unsigned long long) * init.size(),
                                    cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) {
      const int64_t blocks = (a.rows + 255) / 256;
      k_alloc_eval<<<(int)blocks, 256, 0, st>>>(a);
      e = cudaGetLastError();
    }
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(init.data(), dev, sizeof(unsigned long long) * init.size(),
                          cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
      err = cuda_fail(e);
      return 0;
    }
    if (pt)
      for (int t = 0; t < nt; ++t) pt[t] = init[1 + t];
    if (vmin)
      for (int j = 0; j + 1 < a.J; ++j) vmin[j] = from_bits((int64_t)init[1 + nt + j]);
    return init[0];
  }
};

}  // namespace
}  // namespace seedq

extern "C" seedq_status seedq_allocate(const seedq_factor_desc *tensors, int32_t count, int32_t J,
                                       const int32_t *S, const int32_t *k, const double *slopes,
                                       double rbar, double floor_f, double *theta, int32_t *j_tie,
                                       double *q_out, int64_t *tie_count, uint64_t *stream_bits,
                                       void *cuda_stream) {
  if (!tensors || count < 1 || count > (1 << 20) || J < 1 || J > kMaxJ || !S || !k ||
      (J > 1 && (!slopes || !theta)) || !j_tie || !q_out || !tie_count || !stream_bits)
    return SEEDQ_ERR_INVALID_ARG;
  if (!(rbar > 0.0) || !(floor_f >= 0.0) || !(floor_f <= 1.0)) return SEEDQ_ERR_INVALID_ARG;
  int32_t L[kMaxJ] = {0};
  for (int j = 0; j < J; ++j) {
    if (!rung_supported(S[j], k[j])) return SEEDQ_ERR_UNSUPPORTED;
    L[j] = S[j] + 4 * k[j] + 4;
    if (j > 0 && L[j] <= L[j - 1]) return SEEDQ_ERR_SCHEDULE;
  }
  for (int j = 0; j + 1 < J; ++j)
    if (!(slopes[j] > 0.0) || !isfinite(slopes[j])) return SEEDQ_ERR_SCHEDULE;
  uint64_t nblocks = 0;
  for (int t = 0; t < count; ++t) {
    const seedq_factor_desc &d = tensors[t];
    if (d.rows < 1 || d.rows > (1ll << 24) || d.cols < 8 || d.cols % 8 || d.cols > kMaxCols || !d.a)
      return SEEDQ_ERR_INVALID_ARG;
    double asum = 0.0;
    for (int64_t c = 0; c < d.cols; ++c) {
      if (!isfinite(d.a[c]) || d.a[c] < 0.f) return SEEDQ_ERR_INVALID_ARG;
      asum += d.a[c];
    }
    if (!(asum > 0.0)) return SEEDQ_ERR_INVALID_ARG;
    if (d.rho)
      for (int64_t r = 0; r < d.rows; ++r)
        if (!isfinite(d.rho[r]) || !(d.rho[r] > 0.f)) return SEEDQ_ERR_INVALID_ARG;
    nblocks += (uint64_t)d.rows * (uint64_t)(d.cols / 8);
  }
  cudaStream_t st = (cudaStream_t)cuda_stream;

  // Factors of every tensor, exactly as the plan computes them: one device
  // allocation, one upload of all a and rho, three launches for all tensors.
  std::vector<void *> owned;
  auto cleanup = [&]() {
    for (void *p : owned) cudaFree(p);
  };
  auto dalloc = [&](size_t bytes) -> void * {
    void *p = nullptr;
    if (cudaMalloc(&p, bytes) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    owned.push_back(p);
    return p;
  };
  int64_t n_a = 0, n_rho = 0, n_rows = 0, n_nb = 0;
  for (int t = 0; t < count; ++t) {
    n_a += tensors[t].cols;
    n_rho += tensors[t].rho ? tensors[t].rows : 0;
    n_rows += tensors[t].rows;
    n_nb += tensors[t].cols / 8;
  }
  std::vector<float> h_in((size_t)(n_a + n_rho));
  float *d_in = (float *)dalloc(sizeof(float) * (size_t)(n_a + n_rho));
  int32_t *d_perm = (int32_t *)dalloc(sizeof(int32_t) * (size_t)n_a);
  double *d_abar = (double *)dalloc(sizeof(double) * (size_t)n_nb);
  double *d_rho = (double *)dalloc(sizeof(double) * (size_t)n_rows);
  FacJob *d_jobs = (FacJob *)dalloc(sizeof(FacJob) * count);
  // Stable column rankings of all tensors in one sort and one rank launch.
  float *d_skey = (float *)dalloc(sizeof(float) * (size_t)n_a);
  int32_t *d_sidx = (int32_t *)dalloc(sizeof(int32_t) * (size_t)n_a);
  RankJob<float> *d_rjobs = (RankJob<float> *)dalloc(sizeof(RankJob<float>) * count);
  std::vector<RankJob<float>> hr(count);
  if (!d_in || !d_perm || !d_abar || !d_rho || !d_jobs || !d_skey || !d_sidx || !d_rjobs) {
    cleanup();
    return SEEDQ_ERR_NOMEM;
  }
  std::vector<FacJob> hj(count);
  std::vector<AllocTensor> ht(count);
  int64_t rows_total = 0;
  {
    int64_t oa = 0, orh = n_a, orow = 0, onb = 0;
    for (int t = 0; t < count; ++t) {
      const seedq_factor_desc &d = tensors[t];
      memcpy(h_in.data() + oa, d.a, sizeof(float) * d.cols);
      const float *rho_dev = nullptr;
      if (d.rho) {
        memcpy(h_in.data() + orh, d.rho, sizeof(float) * d.rows);
        rho_dev = d_in + orh;
        orh += d.rows;
      }
      hj[t] = FacJob{d_in + oa, rho_dev, d_perm + oa, d_abar + onb, d_rho + orow, d.rows,
                     (int32_t)d.cols};
      hr[t] = RankJob<float>{d_in + oa, d_perm + oa, d_skey + oa, d_sidx + oa, (int32_t)d.cols, 0, 0};
      ht[t] = AllocTensor{d_abar + onb, d_rho + orow, d.rows, rows_total, d.rho ? (int32_t)d.rows : 1,
                          (int32_t)(d.cols / 8)};
      rows_total += ht[t].nrows;
      oa += d.cols;
      orow += d.rows;
      onb += d.cols / 8;
    }
  }
  {
    cudaError_t e = cudaMemcpyAsync(d_in, h_in.data(), sizeof(float) * h_in.size(),
                                    cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(d_jobs, hj.data(), sizeof(FacJob) * count, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = launch_rank<float, false>(hr.data(), count, d_rjobs, st);
    if (e == cudaSuccess) {
      k_factors_multi<<<count, 1024, 0, st>>>(d_jobs);
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // h_in is pageable and goes out of scope
    if (e != cudaSuccess) {
      cleanup();
      return cuda_fail(e);
    }
  }
  AllocTensor *dt = (AllocTensor *)dalloc(sizeof(AllocTensor) * count);
  unsigned long long *dev = (unsigned long long *)dalloc(sizeof(unsigned long long) * (1 + count + kMaxJ));
  if (!dt || !dev) {
    cleanup();
    return SEEDQ_ERR_NOMEM;
  }
  {
    const cudaError_t e =
        cudaMemcpyAsync(dt, ht.data(), sizeof(AllocTensor) * count, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) {
      cleanup();
      return cuda_fail(e);
    }
  }
  Allocator A;
  memset(&A.base, 0, sizeof A.base);
  A.base.t = dt;
  A.base.nt = count;
  A.base.rows = rows_total;
  A.base.J = J;
  for (int j = 0; j < J; ++j) A.base.L[j] = L[j];
  A.st = st;
  A.dev = dev;
  A.nt = count;
  auto thresholds = [&](double lambda, double *th) {
    for (int j = 0; j + 1 < J; ++j) th[j] = lambda / slopes[j];
  };
  auto finish = [&](seedq_status rc) {
    cleanup();
    return A.err != SEEDQ_OK ? A.err : rc;
  };

  // Floor: the m-th smallest raw importance, m = ceil(f N) (positive doubles
  // order as their bit patterns).
  uint64_t m = (uint64_t)ceil(floor_f * (double)nblocks);
  if (m < 1) m = 1;
  int64_t lo = 0, hi = to_bits(INFINITY);
  while (lo < hi && A.err == SEEDQ_OK) {
    const int64_t mid = lo + (hi - lo) / 2;
    if (A.run(kCountLE, 0.0, from_bits(mid), nullptr) >= m) hi = mid;
    else lo = mid + 1;
  }
  const double q = from_bits(lo);
  *q_out = q;

  // Multiplier: bisection on lambda for payload bits <= floor(8 rbar N).
  const uint64_t budget = (uint64_t)floor(8.0 * rbar * (double)nblocks);
  double th_lo[kMaxJ] = {0}, th_hi[kMaxJ] = {0};
  std::vector<uint64_t> pt(count);
  thresholds(INFINITY, th_hi);
  if (A.run(kBits, q, 0.0, th_hi) > budget) return finish(SEEDQ_ERR_SCHEDULE);
  thresholds(0.0, th_lo);
  if (A.run(kBits, q, 0.0, th_lo, pt.data()) <= budget) {  // every block on the top rung
    for (int j = 0; j + 1 < J; ++j) theta[j] = th_lo[j];
    *j_tie = -1;
    for (int t = 0; t < count; ++t) {
      tie_count[t] = 0;
      stream_bits[t] = pt[t];
    }
    return finish(SEEDQ_OK);
  }
  lo = 0;
  hi = to_bits(INFINITY);
  while (hi - lo > 1 && A.err == SEEDQ_OK) {  // bits(lo) > budget >= bits(hi)
    const int64_t mid = lo + (hi - lo) / 2;
    double th[kMaxJ];
    thresholds(from_bits(mid), th);
    if (A.run(kBits, q, 0.0, th) > budget) lo = mid;
    else hi = mid;
  }
  thresholds(from_bits(lo), th_lo);
  thresholds(from_bits(hi), th_hi);

  // The critical tied group: blocks with th_lo[j] <= imp < th_hi[j].
  double vmin[kMaxJ];
  A.run(kVmin, q, 0.0, th_lo, nullptr, vmin);
  int jt = -1;
  double v = 0.0;
  for (int j = 0; j + 1 < J; ++j) {
    if (vmin[j] < th_hi[j]) {
      if (jt >= 0) return finish(SEEDQ_ERR_SCHEDULE);
      jt = j;
      v = vmin[j];
    }
  }
  if (jt < 0) return finish(SEEDQ_ERR_SCHEDULE);
  for (int j = 0; j + 1 < J; ++j) theta[j] = th_hi[j];
  theta[jt] = v;
  const uint64_t b_hi = A.run(kBits, q, 0.0, theta, pt.data());
  const uint64_t step = (uint64_t)(L[jt + 1] - L[jt]);
  const uint64_t excess = b_hi > budget ? b_hi - budget : 0;
  uint64_t T = (excess + step - 1) / step;
  // App. A.5: demote members of the group in block order (tensor order, then
  // row-major within a tensor) until the budget is met.
  std::vector<uint64_t> tied(count, 0);
  if (T) A.run(kTied, q, v, nullptr, tied.data());
  for (int t = 0; t < count; ++t) {
    const uint64_t d = T < tied[t] ? T : tied[t];
    tie_count[t] = (int64_t)d;
    T -= d;
    stream_bits[t] = pt[t] - d * step;
  }
  if (T != 0) return finish(SEEDQ_ERR_SCHEDULE);
  *j_tie = jt;
  return finish(SEEDQ_OK);
}
