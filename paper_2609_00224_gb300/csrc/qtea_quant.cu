// The QTEA quantizer's per-layer steps on the GPU (the step before the GEMV): from full-precision
// weights W [N][K] and the curvature diagonal h = diag(H) [K] to the GEMV's inputs.
//
//  * Salient columns (Sec. 3.2): s_j = max_i W_ij^2 * h_j^2, the s largest (ties: lower column),
//    in ascending order.
//  * Ternary assignment (Sec. 3.1, Eq. 2-3): per row and group, beta = the group mean (0 without the
//    bias option), alpha = mean |W - beta|, refitted `fit_iters` times as the mean |W - beta| over
//    the nonzero codes; T = +1 where W - beta > alpha / 2, -1 where W - beta < -alpha / 2, else 0.
//  * Column-wise rescale refinement (Sec. 3.3, Eq. 6-7): `rescale_iters` rounds of
//    v_j = mean over rows with T_ij != 0 of |W_ij - beta_i| / alpha_i (1 when there are none), then
//    reassignment with the threshold v_j alpha_i / 2.
//  * alpha, beta and v rounded to binary16; the 1:4 residual on each salient column: per group of
//    four rows the row with the largest |W - (alpha v T + beta)| (ties: lower row), its position and
//    the difference in binary16.
// Every value that decides an integer is computed in float32 with the rounding of each operation
// explicit (no contraction into FMA) and every sum in index order, one thread per sum: the results
// are those of the float32 reference bit for bit. The error propagation of Sec. 3.4 is not part of
// these steps.
#include <cuda_fp16.h>

#include <algorithm>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr int kQThreads = 256;

__device__ __forceinline__ int8_t assign(float d, float half) { return d > half ? 1 : (d < -half ? -1 : 0); }

// max_i W_ij * W_ij over a chunk of rows per block row of the grid; the squares are >= 0, so their
// bit patterns order as unsigned integers and the maximum is exact in any order.
constexpr int kQScoreRows = 256;

__global__ void __launch_bounds__(kQThreads) quant_wmax_kernel(const float* __restrict__ W, int N, int K,
                                                              unsigned* __restrict__ wmax) {
  const int j = blockIdx.x * kQThreads + threadIdx.x;
  if (j >= K) return;
  const int i0 = blockIdx.y * kQScoreRows, i1 = min(N, i0 + kQScoreRows);
  float m = 0.f;
  for (int i = i0; i < i1; ++i) {
    const float w = W[(size_t)i * K + j];
    m = fmaxf(m, __fmul_rn(w, w));
  }
  atomicMax(wmax + j, __float_as_uint(m));
}

// s_j = (max_i W_ij^2) * (h_j * h_j).
__global__ void __launch_bounds__(kQThreads) quant_scores_kernel(const unsigned* __restrict__ wmax,
                                                                const float* __restrict__ h, int K,
                                                                float* __restrict__ score) {
  const int j = blockIdx.x * kQThreads + threadIdx.x;
  if (j < K) score[j] = __fmul_rn(__uint_as_float(wmax[j]), __fmul_rn(h[j], h[j]));
}

// flag[j] = 1 when fewer than s columns rank above column j (a higher score, or an equal score and
// a lower index).
constexpr int kQRankThreads = 64;

__global__ void __launch_bounds__(kQRankThreads) quant_rank_kernel(const float* __restrict__ score, int K, int s,
                                                                  int* __restrict__ flag) {
  __shared__ float tile[kQRankThreads];
  const int j = blockIdx.x * kQRankThreads + threadIdx.x;
  const float sj = j < K ? score[j] : 0.f;
  int rank = 0;
  for (int t0 = 0; t0 < K; t0 += kQRankThreads) {
    const int k = t0 + threadIdx.x;
    tile[threadIdx.x] = k < K ? score[k] : 0.f;
    __syncthreads();
    const int n = min(kQRankThreads, K - t0);
    for (int u = 0; u < n; ++u) {
      const float sk = tile[u];
      rank += (sk > sj || (sk == sj && t0 + u < j)) ? 1 : 0;
    }
    __syncthreads();
  }
  if (j < K) flag[j] = rank < s ? 1 : 0;
}

// The flagged columns in ascending order: one block, each thread a contiguous segment.
__global__ void __launch_bounds__(1024) quant_compact_kernel(const int* __restrict__ flag, int K,
                                                            int32_t* __restrict__ sal) {
  __shared__ int cnt[1024];
  const int seg = (K + 1023) / 1024, c0 = threadIdx.x * seg, c1 = min(K, c0 + seg);
  int n = 0;
  for (int c = c0; c < c1; ++c) n += flag[c];
  cnt[threadIdx.x] = n;
  __syncthreads();
  for (int off = 1; off < 1024; off <<= 1) {  // inclusive scan
    const int v = threadIdx.x >= off ? cnt[threadIdx.x - off] : 0;
    __syncthreads();
    cnt[threadIdx.x] += v;
    __syncthreads();
  }
  int pos = cnt[threadIdx.x] - n;
  for (int c = c0; c < c1; ++c)
    if (flag[c]) sal[pos++] = c;
}

// One thread per (row, group) (groups wider than 128 columns): beta, alpha and the codes of the group.
__global__ void __launch_bounds__(kQThreads) quant_group_fit_kernel(const float* __restrict__ W, int N, int K, int group,
                                                                   int G, int bias, int fit_iters,
                                                                   float* __restrict__ alpha, float* __restrict__ beta,
                                                                   int8_t* __restrict__ T) {
  const long long idx = (long long)blockIdx.x * kQThreads + threadIdx.x;
  if (idx >= (long long)N * G) return;
  const int i = (int)(idx / G), gi = (int)(idx - (long long)i * G);
  const int c0 = gi * group, n = min(K, c0 + group) - c0;
  const float* w = W + (size_t)i * K + c0;
  const float fn = (float)n;
  float b = 0.f;
  if (bias) {
    float acc = 0.f;
    for (int c = 0; c < n; ++c) acc = __fadd_rn(acc, w[c]);
    b = __fdiv_rn(acc, fn);
  }
  float acc = 0.f;
  for (int c = 0; c < n; ++c) acc = __fadd_rn(acc, fabsf(__fsub_rn(w[c], b)));
  float a = __fdiv_rn(acc, fn);
  for (int it = 0; it < fit_iters; ++it) {
    const float half = __fmul_rn(a, 0.5f);
    float num = 0.f;
    int cnt = 0;
    for (int c = 0; c < n; ++c) {
      const float d = __fsub_rn(w[c], b);
      if (d > half || d < -half) {
        num = __fadd_rn(num, fabsf(d));
        ++cnt;
      }
    }
    if (cnt > 0) a = __fdiv_rn(num, (float)cnt);
  }
  const float half = __fmul_rn(a, 0.5f);
  int8_t* t = T + (size_t)i * K + c0;
  for (int c = 0; c < n; ++c) t[c] = assign(__fsub_rn(w[c], b), half);
  alpha[idx] = a;
  beta[idx] = b;
}

// Groups of at most 128 columns: one warp per tile of 32 rows x one group. The tile is read into
// shared memory with coalesced loads (row stride 129 words: lane l's row starts in bank l), each lane
// runs its row's passes there in column order, overwrites the tile with its codes, and the codes go
// out with coalesced stores.
constexpr int kQFitWarps = 2;
constexpr int kQFitStride = 129;

__global__ void __launch_bounds__(kQFitWarps * 32) quant_group_fit_tiled_kernel(
    const float* __restrict__ W, int N, int K, int group, int G, int bias, int fit_iters, float* __restrict__ alpha,
    float* __restrict__ beta, int8_t* __restrict__ T) {
  __shared__ float tile[kQFitWarps][32 * kQFitStride];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long t_idx = (long long)blockIdx.x * kQFitWarps + warp;
  const int row_blocks = (N + 31) / 32;
  if (t_idx >= (long long)row_blocks * G) return;
  const int rb = (int)(t_idx / G), gi = (int)(t_idx - (long long)rb * G);
  const int c0 = gi * group, n = min(K, c0 + group) - c0;
  float* tl = tile[warp];
  for (int r0 = 0; r0 < 32; r0 += 8) {
    float vals[8][4];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const int i = rb * 32 + r0 + r;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int c = lane + 32 * k;
        vals[r][k] = (i < N && c < n) ? W[(size_t)i * K + c0 + c] : 0.f;
      }
    }
#pragma unroll
    for (int r = 0; r < 8; ++r)
#pragma unroll
      for (int k = 0; k < 4; ++k) tl[(r0 + r) * kQFitStride + lane + 32 * k] = vals[r][k];
  }
  __syncwarp();
  const int i = rb * 32 + lane;
  const float* w = tl + lane * kQFitStride;
  const float fn = (float)n;
  float b = 0.f;
  if (bias) {
    float acc = 0.f;
    for (int c = 0; c < n; ++c) acc = __fadd_rn(acc, w[c]);
    b = __fdiv_rn(acc, fn);
  }
  float acc = 0.f;
  for (int c = 0; c < n; ++c) acc = __fadd_rn(acc, fabsf(__fsub_rn(w[c], b)));
  float a = __fdiv_rn(acc, fn);
  for (int it = 0; it < fit_iters; ++it) {
    const float half = __fmul_rn(a, 0.5f);
    float num = 0.f;
    int cnt = 0;
    for (int c = 0; c < n; ++c) {
      const float d = __fsub_rn(w[c], b);
      if (d > half || d < -half) {
        num = __fadd_rn(num, fabsf(d));
        ++cnt;
      }
    }
    if (cnt > 0) a = __fdiv_rn(num, (float)cnt);
  }
  const float half = __fmul_rn(a, 0.5f);
  float* wt = tl + lane * kQFitStride;
  for (int c = 0; c < n; ++c) wt[c] = (float)assign(__fsub_rn(wt[c], b), half);
  if (i < N) {
    alpha[(size_t)i * G + gi] = a;
    beta[(size_t)i * G + gi] = b;
  }
  __syncwarp();
  for (int r = 0; r < 32; ++r) {
    const int ii = rb * 32 + r;
    if (ii >= N) break;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int c = lane + 32 * k;
      if (c < n) T[(size_t)ii * K + c0 + c] = (int8_t)tl[r * kQFitStride + c];
    }
  }
}


__global__ void quant_fill_kernel(float* __restrict__ v, int K) {
  const int j = blockIdx.x * kQThreads + threadIdx.x;
  if (j < K) v[j] = 1.f;
}

// v_j = (sum over rows with T_ij != 0, in row order, of |W_ij - beta| / alpha) / count, kept when the
// count is 0. One CTA per 32 columns: warps 1..7 stage the terms of 128-row tiles in shared memory
// (a marker word where T_ij = 0), double-buffered, while warp 0 adds the previous tile in row order.
constexpr int kQSumWarps = 8;
constexpr int kQSumRows = 128;
constexpr unsigned kQNoTerm = 0xFFFFFFFFu;  // a NaN that no division here produces

__global__ void __launch_bounds__(kQSumWarps * 32) quant_colsum_kernel(const float* __restrict__ W,
                                                                      const float* __restrict__ alpha,
                                                                      const float* __restrict__ beta,
                                                                      const int8_t* __restrict__ T, int N, int K,
                                                                      int group, int G, float* __restrict__ v) {
  __shared__ unsigned buf[2][kQSumRows][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.x * 32 + lane;
  const bool jin = j < K;
  const int g = jin ? j / group : 0;
  const int n_tiles = (N + kQSumRows - 1) / kQSumRows;
  float acc = 0.f;
  int cnt = 0;
  for (int k = 0; k <= n_tiles; ++k) {
    if (warp == 0) {
      if (k > 0) {
        const unsigned(*tb)[32] = buf[(k - 1) & 1];
        const int rows = min(kQSumRows, N - (k - 1) * kQSumRows);  // rows past N hold the marker
        for (int r0 = 0; r0 < rows; r0 += 8) {
          unsigned u[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) u[q] = tb[r0 + q][lane];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            if (u[q] != kQNoTerm) {
              acc = __fadd_rn(acc, __uint_as_float(u[q]));
              ++cnt;
            }
          }
        }
      }
    } else if (k < n_tiles) {
      // warp w (1..7) takes rows w - 1, w + 6, ... of the tile: all its loads issued before any term
      unsigned(*tb)[32] = buf[k & 1];
      const int i0 = k * kQSumRows;
      constexpr int kPer = (kQSumRows + kQSumWarps - 2) / (kQSumWarps - 1);
      int8_t t[kPer];
      float w[kPer], al[kPer], be[kPer];
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        const int r = warp - 1 + q * (kQSumWarps - 1), i = i0 + r;
        const bool in = r < kQSumRows && i < N && jin;
        t[q] = in ? T[(size_t)i * K + j] : (int8_t)0;
        w[q] = in ? W[(size_t)i * K + j] : 0.f;
        al[q] = in ? alpha[(size_t)i * G + g] : 1.f;
        be[q] = in ? beta[(size_t)i * G + g] : 0.f;
      }
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        const int r = warp - 1 + q * (kQSumWarps - 1);
        if (r < kQSumRows)
          tb[r][lane] = t[q] != 0 ? __float_as_uint(__fdiv_rn(fabsf(__fsub_rn(w[q], be[q])), al[q])) : kQNoTerm;
      }
    }
    __syncthreads();
  }
  if (warp == 0 && jin && cnt > 0) v[j] = __fdiv_rn(acc, (float)cnt);
}

// The same column sums with the tiles streamed: 16-byte rows (K % 16 == 0), so W, the codes and
// alpha, beta of a 128-row tile reach shared memory by cp.async, four tiles in flight. Warps 1..31
// turn a landed tile into terms (the marker where T_ij = 0) while warp 0 adds the previous tile's
// terms in row order.
constexpr int kCsStages = 4;
constexpr int kCsWarps = 32;  // warp 0 adds; 31 warps form the terms (the divisions bound them)

struct CsSmem {
  float w[kCsStages][kQSumRows][32];
  int8_t t[kCsStages][kQSumRows][32];
  float ab[kCsStages][kQSumRows][2];
  unsigned term[2][kQSumRows][32];
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}

__global__ void __launch_bounds__(kCsWarps * 32) quant_colsum_async_kernel(const float* __restrict__ W,
                                                                            const float* __restrict__ alpha,
                                                                            const float* __restrict__ beta,
                                                                            const int8_t* __restrict__ T, int N,
                                                                            int K, int group, int G,
                                                                            float* __restrict__ v) {
  extern __shared__ __align__(16) unsigned char cs_raw[];
  CsSmem& sm = *reinterpret_cast<CsSmem*>(cs_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j0 = blockIdx.x * 32;  // 32 columns of one scale group (groups are K or 128 columns)
  const int g = j0 / group;
  const int n_tiles = (N + kQSumRows - 1) / kQSumRows;
  const int pt = threadIdx.x - 32, n_pt = (kCsWarps - 1) * 32;
  auto issue = [&](int k) {
    if (k < n_tiles) {
      const int st = k % kCsStages, i0 = k * kQSumRows;
      for (int c = pt; c < kQSumRows * 8; c += n_pt) {
        const int r = c >> 3, q = c & 7;
        // K % 16 == 0: a 16-byte chunk lies wholly inside or wholly past the row's end
        if (i0 + r < N && j0 + 4 * q < K) cp_async16(&sm.w[st][r][4 * q], W + (size_t)(i0 + r) * K + j0 + 4 * q);
      }
      for (int c = pt; c < kQSumRows * 2; c += n_pt) {
        const int r = c >> 1, q = c & 1;
        if (i0 + r < N && j0 + 16 * q < K) cp_async16(&sm.t[st][r][16 * q], T + (size_t)(i0 + r) * K + j0 + 16 * q);
      }
      for (int r = pt; r < kQSumRows; r += n_pt)
        if (i0 + r < N) {
          cp_async4(&sm.ab[st][r][0], alpha + (size_t)(i0 + r) * G + g);
          cp_async4(&sm.ab[st][r][1], beta + (size_t)(i0 + r) * G + g);
        }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  if (warp > 0)
    for (int k = 0; k < kCsStages - 1; ++k) issue(k);
  float acc = 0.f;
  int cnt = 0;
  for (int k = 0; k <= n_tiles; ++k) {
    if (warp > 0) {
      if (k < n_tiles) {
        issue(k + kCsStages - 1);
        asm volatile("cp.async.wait_group %0;" ::"n"(kCsStages - 1) : "memory");
        asm volatile("bar.sync 1, %0;" ::"r"(n_pt) : "memory");  // every producer's copies of tile k
        const int st = k % kCsStages, i0 = k * kQSumRows;
        unsigned(*tb)[32] = sm.term[k & 1];
        for (int e = pt; e < kQSumRows * 32; e += n_pt) {
          const int r = e >> 5, c = e & 31;
          unsigned u = kQNoTerm;
          if (i0 + r < N && j0 + c < K && sm.t[st][r][c] != 0)
            u = __float_as_uint(__fdiv_rn(fabsf(__fsub_rn(sm.w[st][r][c], sm.ab[st][r][1])), sm.ab[st][r][0]));
          tb[r][c] = u;
        }
      }
    } else if (k > 0) {
      const unsigned(*tb)[32] = sm.term[(k - 1) & 1];
      const int rows = min(kQSumRows, N - (k - 1) * kQSumRows);  // rows past N hold the marker
      for (int r0 = 0; r0 < rows; r0 += 8) {
        unsigned u[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) u[q] = tb[r0 + q][lane];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (u[q] != kQNoTerm) {
            acc = __fadd_rn(acc, __uint_as_float(u[q]));
            ++cnt;
          }
        }
      }
    }
    __syncthreads();
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  if (warp == 0 && j0 + lane < K && cnt > 0) v[j0 + lane] = __fdiv_rn(acc, (float)cnt);
}

// T_ij = nearest of {-v_j alpha, 0, +v_j alpha} to W_ij - beta (threshold (v_j alpha) / 2), every entry.
// With K % 4 == 0 a thread takes four columns of one row (one 16-byte load of W, one 4-byte store of
// codes; the four columns share a scale group); otherwise one entry.
template <bool VEC>
__global__ void __launch_bounds__(kQThreads) quant_reassign_kernel(const float* __restrict__ W,
                                                                  const float* __restrict__ alpha,
                                                                  const float* __restrict__ beta,
                                                                  const float* __restrict__ v, int N, int K,
                                                                  int group, int G, int8_t* __restrict__ T) {
  const int per = VEC ? 4 : 1;
  const int j = (blockIdx.x * kQThreads + threadIdx.x) * per;
  if (j >= K) return;
  for (int i = blockIdx.y; i < N; i += gridDim.y) {
    const size_t e = (size_t)i * K + j, sg = (size_t)i * G + j / group;
    const float al = alpha[sg], be = beta[sg];
    if (VEC) {
      const float4 w = *reinterpret_cast<const float4*>(W + e);
      const float4 vv = *reinterpret_cast<const float4*>(v + j);
      const float wv[4] = {w.x, w.y, w.z, w.w}, vj[4] = {vv.x, vv.y, vv.z, vv.w};
      uint32_t packed = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q)
        packed |= (uint32_t)(uint8_t)assign(__fsub_rn(wv[q], be), __fmul_rn(__fmul_rn(vj[q], al), 0.5f)) << (8 * q);
      *reinterpret_cast<uint32_t*>(T + e) = packed;
    } else {
      T[e] = assign(__fsub_rn(W[e], be), __fmul_rn(__fmul_rn(v[j], al), 0.5f));
    }
  }
}

// alpha, beta (pairs with bias) and v in binary16.
__global__ void __launch_bounds__(kQThreads) quant_round_kernel(const float* __restrict__ alpha, const float* __restrict__ beta,
                                                               const float* __restrict__ v, long long NG, int K, int bias,
                                                               uint16_t* __restrict__ row_scale,
                                                               uint16_t* __restrict__ col_scale) {
  const long long idx = (long long)blockIdx.x * kQThreads + threadIdx.x;
  if (idx < NG) {
    if (bias) {
      row_scale[2 * (size_t)idx] = __half_as_ushort(__float2half_rn(alpha[idx]));
      row_scale[2 * (size_t)idx + 1] = __half_as_ushort(__float2half_rn(beta[idx]));
    } else {
      row_scale[idx] = __half_as_ushort(__float2half_rn(alpha[idx]));
    }
  }
  if (idx < K) col_scale[idx] = __half_as_ushort(__float2half_rn(v[idx]));
}

// One thread per (group of four rows q, byte of positions c4): the residual of salient entries
// 4 c4 .. 4 c4 + 3 against the binary16 alpha, beta and v.
__global__ void __launch_bounds__(kQThreads) quant_residual_kernel(const float* __restrict__ W, const int8_t* __restrict__ T,
                                                                  const uint16_t* __restrict__ row_scale,
                                                                  const uint16_t* __restrict__ col_scale,
                                                                  const int32_t* __restrict__ sal, int N, int K,
                                                                  int group, int G, int s, int bias,
                                                                  uint16_t* __restrict__ rvals,
                                                                  uint8_t* __restrict__ ridx) {
  const int nb = (s + 3) / 4;
  const long long idx = (long long)blockIdx.x * kQThreads + threadIdx.x;
  if (idx >= (long long)(N / 4) * nb) return;
  const int q = (int)(idx / nb), c4 = (int)(idx - (long long)q * nb);
  uint32_t byte = 0;
  for (int k = 0; k < 4; ++k) {
    const int c = 4 * c4 + k;
    if (c >= s) break;
    const int j = sal[c], g = j / group;
    const float vj = __half2float(__ushort_as_half(col_scale[j]));
    int best = 0;
    float best_abs = -1.f, best_r = 0.f;
    for (int p = 0; p < 4; ++p) {
      const int i = 4 * q + p;
      const size_t e = (size_t)i * G + g;
      const float a = __half2float(__ushort_as_half(bias ? row_scale[2 * e] : row_scale[e]));
      const float b = bias ? __half2float(__ushort_as_half(row_scale[2 * e + 1])) : 0.f;
      const float what = __fadd_rn(__fmul_rn(__fmul_rn(a, vj), (float)T[(size_t)i * K + j]), b);
      const float r = __fsub_rn(W[(size_t)i * K + j], what);
      if (fabsf(r) > best_abs) {
        best_abs = fabsf(r);
        best = p;
        best_r = r;
      }
    }
    rvals[(size_t)q * s + c] = __half_as_ushort(__float2half_rn(best_r));
    byte |= (uint32_t)best << (2 * k);
  }
  ridx[(size_t)q * nb + c4] = (uint8_t)byte;
}

inline unsigned blocks(long long n, int per) { return (unsigned)((n + per - 1) / per); }

// The streamed column-sum kernel's shared memory is above the default 48 KB: opt in once.
bool cs_async_ready() {
  static const bool ready = [] {  // initialised once, thread-safe
    const bool ok = cudaFuncSetAttribute(quant_colsum_async_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)sizeof(CsSmem)) == cudaSuccess;
    if (!ok) cudaGetLastError();
    return ok;
  }();
  return ready;
}

}  // namespace

cudaError_t launch_quantize(const QuantArgs& a, cudaStream_t st) {
  const int G = (a.K + a.group - 1) / a.group;
  const long long NG = (long long)a.N * G;
  // scratch: wmax [K], score [K], flag [K], v [K], alpha [N][G], beta [N][G], all 4-byte words
  char* scratch = nullptr;
  const size_t words = 4 * (size_t)a.K + 2 * (size_t)NG;
  cudaError_t e = cudaMallocAsync(&scratch, 4 * words, st);
  if (e != cudaSuccess) return e;
  unsigned* wmax = reinterpret_cast<unsigned*>(scratch);
  float* score = reinterpret_cast<float*>(wmax + a.K);
  int* flag = reinterpret_cast<int*>(score + a.K);
  float* v = reinterpret_cast<float*>(flag + a.K);
  float* alpha = v + a.K;
  float* beta = alpha + NG;
  const unsigned kb = blocks(a.K, kQThreads);
  if (a.s > 0) {
    e = cudaMemsetAsync(wmax, 0, sizeof(unsigned) * (size_t)a.K, st);
    if (e == cudaSuccess) {
      quant_wmax_kernel<<<dim3(kb, blocks(a.N, kQScoreRows)), kQThreads, 0, st>>>(a.W, a.N, a.K, wmax);
      quant_scores_kernel<<<kb, kQThreads, 0, st>>>(wmax, a.h, a.K, score);
      quant_rank_kernel<<<blocks(a.K, kQRankThreads), kQRankThreads, 0, st>>>(score, a.K, a.s, flag);
      quant_compact_kernel<<<1, 1024, 0, st>>>(flag, a.K, a.sal);
    }
  }
  if (e == cudaSuccess) {
    if (a.group <= 128)
      quant_group_fit_tiled_kernel<<<blocks((long long)((a.N + 31) / 32) * G, kQFitWarps), kQFitWarps * 32, 0, st>>>(
          a.W, a.N, a.K, a.group, G, a.bias, a.fit_iters, alpha, beta, a.codes);
    else
      quant_group_fit_kernel<<<blocks(NG, kQThreads), kQThreads, 0, st>>>(a.W, a.N, a.K, a.group, G, a.bias,
                                                                          a.fit_iters, alpha, beta, a.codes);
    quant_fill_kernel<<<kb, kQThreads, 0, st>>>(v, a.K);
    // with K % 4 == 0 every row of W (16-byte aligned base), of the codes (4-byte aligned base) and
    // the v scratch (3K words into the allocation) keep those alignments
    const bool vec = a.K % 4 == 0 && (reinterpret_cast<uintptr_t>(a.W) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(a.codes) & 3) == 0;
    const dim3 rgrid(blocks(vec ? a.K / 4 : a.K, kQThreads), (unsigned)std::min(a.N, 65535));
    // streamed column sums where every row of W and of the codes is 16-byte aligned
    const bool cs_async = a.K % 16 == 0 && (reinterpret_cast<uintptr_t>(a.W) & 15) == 0 &&
                          (reinterpret_cast<uintptr_t>(a.codes) & 15) == 0 && cs_async_ready();
    for (int it = 0; it < a.rescale_iters; ++it) {
      if (cs_async)
        quant_colsum_async_kernel<<<blocks(a.K, 32), kCsWarps * 32, sizeof(CsSmem), st>>>(
            a.W, alpha, beta, a.codes, a.N, a.K, a.group, G, v);
      else
        quant_colsum_kernel<<<blocks(a.K, 32), kQSumWarps * 32, 0, st>>>(a.W, alpha, beta, a.codes, a.N, a.K,
                                                                          a.group, G, v);
      if (vec)
        quant_reassign_kernel<true><<<rgrid, kQThreads, 0, st>>>(a.W, alpha, beta, v, a.N, a.K, a.group, G, a.codes);
      else
        quant_reassign_kernel<false><<<rgrid, kQThreads, 0, st>>>(a.W, alpha, beta, v, a.N, a.K, a.group, G, a.codes);
    }
    quant_round_kernel<<<blocks(NG > a.K ? NG : a.K, kQThreads), kQThreads, 0, st>>>(alpha, beta, v, NG, a.K, a.bias,
                                                                                     a.row_scale, a.col_scale);
    if (a.s > 0)
      quant_residual_kernel<<<blocks((long long)(a.N / 4) * ((a.s + 3) / 4), kQThreads), kQThreads, 0, st>>>(
          a.W, a.codes, a.row_scale, a.col_scale, a.sal, a.N, a.K, a.group, G, a.s, a.bias, a.rvals, a.ridx);
    e = cudaGetLastError();
  }
  const cudaError_t f = cudaFreeAsync(scratch, st);
  return e != cudaSuccess ? e : f;
}

}  // namespace qtea
