// Data-free importance (Sec. 3.2, Eq. gamma, Eq. prop, the backward proxy of
// App. A.1) and the outlier-column statistics and selection (Sec. 3.5,
// App. A.6) over an FP16 checkpoint resident on the device.
//
// Every weight matrix is read once.  One column pass per matrix computes, for
// a tile of 32 input columns over all rows:
//   * the weighted column sums of squares sum_r W_rc^2 g_r of the backward
//     proxy (g the residual-gradient scale the matrix writes to),
//   * the partial row sums of squares sum_{c in tile} W_rc^2 a_c of Eq. prop
//     (for W_v, W_gate, W_up),
//   * the column maximum of |W| and a 256-bin histogram of the top eight bits
//     of |W| (exponent and three mantissa bits) per column, which bounds the
//     column median from below; columns whose dynamic range could reach the
//     threshold get their exact median from a second sweep of the tile that
//     histograms the low seven bits inside the median's bins.
// Layers are taken in reverse order because each layer's column sums need the
// stream scale left by the layer above; a small kernel per step finishes the
// stream update, rho, a^(down) (Gauss-Hermite) and a^(o) (repeat_kv).
//
// Arithmetic: squares of FP16 values are exact in fp32; each product with the
// fp32-rounded weight is rounded once, chunks of 16 rows accumulate in fp32
// and then in fp64, partial row sums of 32 columns are fp32, their tile sums
// fp64; the stream scale G stays fp64.  Tables are rounded to float32 (App.
// A.7).  The outlier statistics are exact: maxima and medians are FP16 values,
// the ratio is one IEEE division of their fp64 sum, the activation mean an
// fp64 sum in column order.
#include <cuda_fp16.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "seedq_internal.cuh"
#include "synth.cuh"

namespace seedq {
namespace {

constexpr int kTC = 32;             // columns per tile
constexpr int kCT = 256;            // threads per CTA of the column pass
constexpr int kPhases = kCT / 4;    // rows per sweep (4 threads x 8 columns per row)
constexpr int kUnroll = 8;          // rows in flight per thread
constexpr int kChunk = 16;          // fp32 accumulation before each fp64 add
constexpr int kHS = 257;            // histogram row stride (bank spread)
constexpr int kGH = 64;             // Gauss-Hermite nodes
constexpr int kMaxJobs = 4;
constexpr double kEpsDR = 5.9604644775390625e-08;  // 2^-24
constexpr double kDrMin = 1.0e3;
constexpr double kActMin = 1.0e2;

__constant__ double c_gh_x[kGH];  // nodes
__constant__ double c_gh_w[kGH];  // weights / sqrt(pi)

struct Cand {
  double v;
  int32_t t, c;
};

struct ColJob {
  const uint16_t *W;
  int64_t R;
  int32_t C;
  int32_t tile0;         // first CTA of this job in the launch
  int32_t g_mode;        // 0 none, 1 all ones, 2 gd[r], 3 gf[r], 4 sum of gd over n_rep heads
  int32_t n_rep, head_dim;
  const double *gd;
  const int *gexp;       // mode 2: gd is scaled by 2^-(*gexp) before use (nullptr: 1)
  const float *gf;
  double *colsum;        // C
  const float *a;        // C, or nullptr (no row partials)
  float *rowpart;        // (C / 32) x R
  double *dr;            // C, or nullptr
  int32_t tensor;        // model order, for the candidate list
  Cand *cand;            // dynamic-range candidates (nullptr: none kept)
  uint32_t *ncand;
};

struct ColArgs {
  ColJob j[kMaxJobs];
  int32_t njobs;
};

__device__ __forceinline__ uint4 ld_stream16(const void *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ double half_mag(uint32_t bits) {
  return (double)__half2float(__ushort_as_half((unsigned short)bits));
}

__device__ __forceinline__ float row_weight(const ColJob &J, int64_t r) {
  switch (J.g_mode) {
    case 1: return 1.f;
    case 2: return (float)(J.gexp ? scalbn(J.gd[r], -*J.gexp) : J.gd[r]);
    case 3: return J.gf[r];
    case 4: {
      // Value-head row r = (key-value head j, offset i) collects the query
      // heads j * n_rep .. j * n_rep + n_rep - 1 at offset i.
      const int j = (int)r / J.head_dim, i = (int)r - j * J.head_dim;
      double s = 0.0;
      for (int k = 0; k < J.n_rep; ++k) s += J.gd[(int64_t)(j * J.n_rep + k) * J.head_dim + i];
      return (float)s;
    }
    default: return 0.f;
  }
}

template <bool kCols, bool kRows>
__device__ __forceinline__ void sweep(const ColJob &J, int tile, uint32_t *hist, float (&av)[8],
                                      double (&cs)[8], uint32_t (&mx)[4]) {
  const int t = threadIdx.x, cg = t & 3, rp = t >> 2;
  const int lane = t & 31;
  const unsigned quad = 0xFu << (lane & 28);
  const int lc0 = cg * 8;
  const int64_t R = J.R, C = J.C;
  const uint16_t *base = J.W + (int64_t)tile * kTC + lc0;
  float cf[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) cf[q] = 0.f;
  int nchunk = 0;
  for (int64_t r0 = rp; r0 < R; r0 += (int64_t)kUnroll * kPhases) {
    uint4 w[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t r = r0 + (int64_t)u * kPhases;
      w[u] = r < R ? ld_stream16(base + r * C) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t r = r0 + (int64_t)u * kPhases;
      if (r >= R) break;
      const float gr = kCols ? row_weight(J, r) : 0.f;
      const uint32_t wd[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
      float rs = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t m = wd[q] & 0x7fff7fffu;
        mx[q] = __vmaxu2(mx[q], m);
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&wd[q]));
        const float s0 = f.x * f.x, s1 = f.y * f.y;
        if (kCols) {
          cf[2 * q] = fmaf(s0, gr, cf[2 * q]);
          cf[2 * q + 1] = fmaf(s1, gr, cf[2 * q + 1]);
        }
        if (kRows) {
          rs = fmaf(s0, av[2 * q], rs);
          rs = fmaf(s1, av[2 * q + 1], rs);
        }
        atomicAdd(hist + (lc0 + 2 * q) * kHS + ((m >> 7) & 0xffu), 1u);
        atomicAdd(hist + (lc0 + 2 * q + 1) * kHS + (m >> 23), 1u);
      }
      if (kRows) {
        rs += __shfl_xor_sync(quad, rs, 1);
        rs += __shfl_xor_sync(quad, rs, 2);
        if (cg == 0) J.rowpart[(int64_t)tile * R + r] = rs;
      }
      if (kCols && ++nchunk == kChunk) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          cs[q] += (double)cf[q];
          cf[q] = 0.f;
        }
        nchunk = 0;
      }
    }
  }
  if (kCols) {
#pragma unroll
    for (int q = 0; q < 8; ++q) cs[q] += (double)cf[q];
  }
}

__global__ void __launch_bounds__(kCT, 2) k_colpass(const __grid_constant__ ColArgs A) {
  __shared__ __align__(16) uint32_t hist[kTC * kHS];
  __shared__ uint32_t s_b[2][kTC], s_below[2][kTC], s_max[kTC];
  __shared__ int s_need[kTC];
  __shared__ int s_any;
  int ji = 0;
  while (ji + 1 < A.njobs && (int)blockIdx.x >= A.j[ji + 1].tile0) ++ji;
  const ColJob &J = A.j[ji];
  const int tile = (int)blockIdx.x - J.tile0;
  const int t = threadIdx.x, cg = t & 3, rp = t >> 2, lc0 = cg * 8;
  const int64_t R = J.R;
  for (int i = t; i < kTC * kHS; i += kCT) hist[i] = 0u;
  if (t == 0) s_any = 0;
  float av[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) av[q] = J.a ? J.a[(int64_t)tile * kTC + lc0 + q] : 0.f;
  double cs[8];
  uint32_t mx[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (int q = 0; q < 8; ++q) cs[q] = 0.0;
  __syncthreads();
  const bool cols = J.g_mode != 0, rows = J.a != nullptr;
  if (cols && rows) sweep<true, true>(J, tile, hist, av, cs, mx);
  else if (cols) sweep<true, false>(J, tile, hist, av, cs, mx);
  else if (rows) sweep<false, true>(J, tile, hist, av, cs, mx);
  else sweep<false, false>(J, tile, hist, av, cs, mx);
  __syncthreads();

  // Bins holding the order statistics k0 = (R-1)/2 and k1 = R/2 of |W|.
  const uint32_t k0 = (uint32_t)((R - 1) / 2), k1 = (uint32_t)(R / 2);
  if (t < kTC) {
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

  // Column sums: fp64 partials of the 64 row phases added in phase order.
  double *red = reinterpret_cast<double *>(hist);
  if (cols) {
#pragma unroll
    for (int q = 0; q < 8; ++q) red[rp * kTC + lc0 + q] = cs[q];
  }
  __syncthreads();
  if (cols && t < kTC) {
    double s = 0.0;
    for (int p = 0; p < kPhases; ++p) s += red[p * kTC + t];
    J.colsum[(int64_t)tile * kTC + t] = s;
  }
  __syncthreads();
  uint32_t *rmx = hist;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    rmx[rp * kTC + lc0 + 2 * q] = mx[q] & 0xffffu;
    rmx[rp * kTC + lc0 + 2 * q + 1] = mx[q] >> 16;
  }
  __syncthreads();
  const int64_t col = (int64_t)tile * kTC + t;
  if (t < kTC) {
    uint32_t m = 0;
    for (int p = 0; p < kPhases; ++p) m = max(m, rmx[p * kTC + t]);
    s_max[t] = m;
    // median >= lower edge of bin b0, and x -> max / (x + eps) is monotone
    // under round-to-nearest, so this bounds the rounded statistic.
    const double hi = __ddiv_rn(half_mag(m), __dadd_rn(half_mag(s_b[0][t] << 7), kEpsDR));
    const int need = hi >= kDrMin;
    s_need[t] = need;
    if (need) atomicOr(&s_any, 1);
    else if (J.dr) J.dr[col] = 0.0;
  }
  __syncthreads();
  if (!s_any) return;

  // Exact medians of the columns that may qualify: histogram the low seven
  // bits of the elements in the two median bins.
  uint32_t *h2 = hist;  // kTC x 2 x 128
  for (int i = t; i < kTC * 256; i += kCT) h2[i] = 0u;
  __syncthreads();
  const uint16_t *base = J.W + (int64_t)tile * kTC + lc0;
  for (int64_t r = rp; r < R; r += kPhases) {
    const uint4 w = ld_stream16(base + r * J.C);
    const uint32_t wd[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int lc = lc0 + e;
      if (!s_need[lc]) continue;
      const uint32_t v = (e & 1 ? wd[e >> 1] >> 16 : wd[e >> 1]) & 0x7fffu;
      if ((v >> 7) == s_b[0][lc]) atomicAdd(h2 + lc * 256 + (v & 127u), 1u);
      if ((v >> 7) == s_b[1][lc]) atomicAdd(h2 + lc * 256 + 128 + (v & 127u), 1u);
    }
  }
  __syncthreads();
  if (t < kTC && s_need[t]) {
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
    const double m1 = half_mag((s_b[0][t] << 7) | low[0]);
    const double m2 = half_mag((s_b[1][t] << 7) | low[1]);
    const double med = (m1 + m2) * 0.5;
    const double dr = __ddiv_rn(half_mag(s_max[t]), __dadd_rn(med, kEpsDR));
    const bool keep = dr >= kDrMin;
    if (J.dr) J.dr[col] = keep ? dr : 0.0;
    if (keep && J.cand) {
      const uint32_t slot = atomicAdd(J.ncand, 1u);
      J.cand[slot] = Cand{dr, J.tensor, (int32_t)col};
    }
  }
}

// E[silu(g)^2], g ~ N(0, var), by the Gauss-Hermite rule in constant memory.
__device__ double silu_sq_moment(double var) {
  const double s = sqrt(2.0 * var);
  double acc = 0.0;
  for (int i = 0; i < kGH; ++i) {
    const double g = s * c_gh_x[i];
    const double y = g / (1.0 + exp(-g));
    acc += c_gh_w[i] * (y * y);
  }
  return acc;
}

// Stream-scale bookkeeping.  The backward proxy grows the residual scale by a
// model-dependent factor per layer (tens for Llama shapes), past the float32
// range after a few dozen layers.  Every step therefore works on G scaled by
// an exact power of two: the producer of a new G records the largest binary
// exponent of its entries, and each consumer multiplies by 2^-that exponent
// before rounding to float32.  Scaling by powers of two changes no rounding,
// and rho is stored normalized to unit mean within its tensor, so the scales
// cancel.
struct FinArgs {
  const double *G_old;   // d_model, previous stream scale, or nullptr (head step)
  const int *e_old;      // its exponent
  const double *gx0, *gx1;
  double *G_new;         // d_model
  int *e_new;            // max binary exponent of G_new (atomic max)
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

__global__ void k_fin(const __grid_constant__ FinArgs f) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < f.d) {
    double g = f.G_new[i];
    if (f.G_old) {
      g = scalbn(f.G_old[i], -*f.e_old) + f.gx0[i];
      if (f.gx1) g = g + f.gx1[i];
      f.G_new[i] = g;
    }
    if (g > 0.0) atomicMax(f.e_new, ilogb(g));
    if (f.rho_raw) f.rho_raw[i] = g;
  }
  if (i < f.n_out && f.a_out) {
    if (f.mode == 0) {
      double v = 0.0, u = 0.0;
      for (int t = 0; t < f.ntile; ++t) {
        v += (double)f.rp0[(int64_t)t * f.nrows + i];
        u += (double)f.rp1[(int64_t)t * f.nrows + i];
      }
      f.a_out[i] = (float)(silu_sq_moment(v) * u);
    } else {
      const int h = i / f.head_dim, o = i - h * f.head_dim;
      const int row = (h / f.n_rep) * f.head_dim + o;
      double v = 0.0;
      for (int t = 0; t < f.ntile; ++t) v += (double)f.rp0[(int64_t)t * f.nrows + row];
      f.a_out[i] = (float)v;
    }
  }
}

// rho tables: each vector divided by its mean (summed in row order), float32.
// Block 2l is rho_o of layer l, block 2l + 1 rho_down.
__global__ void k_norm_rho(const double *__restrict__ raw, int d, float *__restrict__ rho_o,
                           float *__restrict__ rho_down) {
  __shared__ double mean;
  const double *v = raw + (int64_t)blockIdx.x * d;
  float *out = ((blockIdx.x & 1) ? rho_down : rho_o) + (int64_t)(blockIdx.x >> 1) * d;
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int i = 0; i < d; ++i) s += v[i];
    mean = s / (double)d;
  }
  __syncthreads();
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

// Activation statistic a_j / mean(a), the mean summed in column order; one
// CTA per tensor.
__global__ void k_act_ratio(const RatioJob *__restrict__ jobs, double *__restrict__ ratio,
                            Cand *__restrict__ cand, uint32_t *__restrict__ ncand) {
  const RatioJob J = jobs[blockIdx.x];
  __shared__ double mean;
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int c = 0; c < J.C; ++c) s += (double)J.a[c];
    mean = s / (double)J.C;
  }
  __syncthreads();
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

int tiles_of(const ColJob &j) { return j.C / kTC; }

seedq_status launch_cols(ColArgs &A, cudaStream_t st) {
  int total = 0;
  for (int i = 0; i < A.njobs; ++i) {
    A.j[i].tile0 = total;
    total += tiles_of(A.j[i]);
  }
  if (total == 0) return SEEDQ_OK;
  k_colpass<<<total, kCT, 0, st>>>(A);
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

struct DevBuf {
  std::vector<void *> ptrs;
  ~DevBuf() {
    for (void *p : ptrs) cudaFree(p);
  }
  template <class T>
  T *get(size_t n, seedq_status *rc) {
    void *p = nullptr;
    if (*rc != SEEDQ_OK) return nullptr;
    const cudaError_t e = cudaMalloc(&p, n * sizeof(T) + 16);
    if (e != cudaSuccess) {
      cudaGetLastError();
      *rc = e == cudaErrorMemoryAllocation ? SEEDQ_ERR_NOMEM : cuda_fail(e);
      return nullptr;
    }
    ptrs.push_back(p);
    return (T *)p;
  }
};

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
  ColArgs A;
  memset(&A, 0, sizeof A);
  A.njobs = 1;
  A.j[0] = stats_job(W, R, (int32_t)C, dyn_range, 0, nullptr, nullptr);
  if (col_sq) {
    A.j[0].g_mode = g ? 3 : 1;
    A.j[0].gf = g;
    A.j[0].colsum = col_sq;
  }
  return launch_cols(A, (cudaStream_t)cuda_stream);
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
  DevBuf B;
  double *Gbuf = B.get<double>((size_t)2 * d, &rc), *gxa = B.get<double>(d, &rc),
         *gxb = B.get<double>(d, &rc);
  double *Gh = B.get<double>(f, &rc), *Ga = B.get<double>(qd, &rc);
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
  double gx[kGH], gw[kGH];
  gauss_hermite(kGH, gx, gw);
  SEEDQ_CUDA(cudaMemcpyToSymbolAsync(c_gh_x, gx, sizeof gx, 0, cudaMemcpyHostToDevice, st));
  SEEDQ_CUDA(cudaMemcpyToSymbolAsync(c_gh_w, gw, sizeof gw, 0, cudaMemcpyHostToDevice, st));
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
  // head, then two per layer) has exponent gexp[s].
  int step = 0;
  auto Gcur = [&]() { return Gbuf + (size_t)(step & 1) * d; };
  auto Gnext = [&]() { return Gbuf + (size_t)((step + 1) & 1) * d; };

  // The head: an isotropic gradient at the logits gives the stream scale.
  {
    ColArgs A;
    memset(&A, 0, sizeof A);
    A.njobs = 1;
    A.j[0] = job(7 * L, m->lm_head);
    A.j[0].g_mode = 1;
    A.j[0].colsum = Gcur();
    if ((rc = launch_cols(A, st)) != SEEDQ_OK) return rc;
    FinArgs F;
    memset(&F, 0, sizeof F);
    F.G_new = Gcur();
    F.e_new = gexp;
    F.rho_raw = rraw + (size_t)(2 * (L - 1) + 1) * d;
    F.d = d;
    k_fin<<<gb, 256, 0, st>>>(F);
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
    A.j[0].g_mode = 2;
    A.j[0].gd = Gcur();
    A.j[0].gexp = gexp + step;
    A.j[0].colsum = Gh;
    if ((rc = launch_cols(A, st)) != SEEDQ_OK) return rc;
    // Gate and up: back-map of Gh, and the row sums of Eq. prop.
    memset(&A, 0, sizeof A);
    A.njobs = 2;
    A.j[0] = job(t0 + 4, y.wgate);
    A.j[1] = job(t0 + 5, y.wup);
    for (int i = 0; i < 2; ++i) {
      A.j[i].g_mode = 2;
      A.j[i].gd = Gh;
      A.j[i].colsum = i ? gxb : gxa;
      A.j[i].a = a_mlp;
      A.j[i].rowpart = i ? rpb : rpa;
    }
    if ((rc = launch_cols(A, st)) != SEEDQ_OK) return rc;
    {
      FinArgs F;
      memset(&F, 0, sizeof F);
      F.G_old = Gcur(); F.e_old = gexp + step; F.gx0 = gxa; F.gx1 = gxb;
      F.G_new = Gnext(); F.e_new = gexp + step + 1;
      F.rho_raw = rraw + (size_t)(2 * l) * d; F.d = d;
      F.rp0 = rpa; F.rp1 = rpb; F.ntile = d / kTC; F.nrows = f;
      F.a_out = out->a_down + (size_t)l * f; F.mode = 0; F.n_out = f;
      k_fin<<<(std::max(d, f) + 255) / 256, 256, 0, st>>>(F);
      SEEDQ_CUDA(cudaGetLastError());
      ++step;
    }
    // Output projection (stream scale in, attention scale out) with the
    // statistics of q and k.
    memset(&A, 0, sizeof A);
    A.njobs = 3;
    A.j[0] = job(t0 + 3, y.wo);
    A.j[0].g_mode = 2;
    A.j[0].gd = Gcur();
    A.j[0].gexp = gexp + step;
    A.j[0].colsum = Ga;
    A.j[1] = job(t0 + 0, y.wq);
    A.j[2] = job(t0 + 1, y.wk);
    if ((rc = launch_cols(A, st)) != SEEDQ_OK) return rc;
    // Value projection: the query heads of each value head summed, and the
    // row sums of a^(o).
    memset(&A, 0, sizeof A);
    A.njobs = 1;
    A.j[0] = job(t0 + 2, y.wv);
    A.j[0].g_mode = 4;
    A.j[0].gd = Ga;
    A.j[0].n_rep = n_rep;
    A.j[0].head_dim = hd;
    A.j[0].colsum = gxa;
    A.j[0].a = a_attn;
    A.j[0].rowpart = rpa;
    if ((rc = launch_cols(A, st)) != SEEDQ_OK) return rc;
    {
      FinArgs F;
      memset(&F, 0, sizeof F);
      F.G_old = Gcur(); F.e_old = gexp + step; F.gx0 = gxa;
      F.G_new = Gnext(); F.e_new = gexp + step + 1;
      F.rho_raw = l > 0 ? rraw + (size_t)(2 * (l - 1) + 1) * d : nullptr; F.d = d;
      F.rp0 = rpa; F.ntile = d / kTC; F.nrows = kvd;
      F.a_out = out->a_o + (size_t)l * qd; F.mode = 1; F.n_out = qd;
      F.n_rep = n_rep; F.head_dim = hd;
      k_fin<<<(std::max(d, qd) + 255) / 256, 256, 0, st>>>(F);
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
