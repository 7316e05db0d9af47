// QTEA GEMV for layouts in the paper's own storage (any batch 1 <= M <= 16):
//
//   y[m][o] = sum_g ( alpha[o][g] sum_{j in g} T[o][j] v[j] x[m][j] + beta[o][g] sum_{j in g} x[m][j] )
//           + sum_{c < s} [pos(o/4, c) == o % 4] R[o/4][c] x[m][S_c]
//
// Eq. 10 in full (Sec. 3.5: alpha and beta per row and group of 128 columns, beta multiplying the
// plain sum of x) plus Eq. 11, with the ternary codes in either this library's 2-bit layout or the
// paper's base-3 layout (five codes per byte, 26 bytes per 128 columns), and residual values in
// fp16 or in the paper's FP8 E4M3.
//
// Three kernels:
//  * qtea_gemv_paper_b3_kernel (base-3, M <= 4): v*x staged once per CTA as fixed point per
//    128-column block, decoded with dp4a through a byte table; several problems per launch.
//  * qtea_gemv_paper_staged_kernel (2-bit, M <= 4): v*x staged once per CTA in fp32.
//  * qtea_gemv_paper_kernel (any layout, any M): one warp per output row reading x and v from
//    global memory. A block lies in one scale group (groups are 128 columns or the whole row);
//    lane l takes code byte l of the block and adds alpha * sum T v x + beta * sum x over its
//    columns for every batch row; the lanes' sums are added once at the end. Base-3 bytes are
//    expanded to five 2-bit codes through a 243-entry table in shared memory. v*x is exact in fp32;
//    sums are fp32.
// In each, the warp of a row adds the residual of the row's group of four.
#include <cuda_fp16.h>

#include <algorithm>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr int kPaperWarps = 4;

template <int MB>
__global__ void __launch_bounds__(kPaperWarps * 32) qtea_gemv_paper_kernel(const PaperParams p) {
  __shared__ uint16_t lut[243];  // base-3 byte -> five 2-bit codes
  for (int i = threadIdx.x; i < 243; i += blockDim.x) {
    int b = i;
    uint32_t v = 0;
    for (int d = 0; d < 5; ++d) {
      v |= (uint32_t)(b % 3) << (2 * d);
      b /= 3;
    }
    lut[i] = (uint16_t)v;
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int o = blockIdx.x * kPaperWarps + warp;
  if (o >= p.N) return;
  const int M = p.M;
  float acc[MB], res[MB];
#pragma unroll
  for (int m = 0; m < MB; ++m) acc[m] = res[m] = 0.f;

  // The row's 128-column blocks in order; within a block lane l takes code byte l (base-3: columns
  // 5l .. 5l+4 for l < 26; 2-bit: columns 4l .. 4l+3), so the warp's loads of codes, x and v are
  // contiguous. alpha and beta of the block's group are the same for every lane.
  const int n_blocks = (p.K + 127) / 128;
  const uint8_t* row = p.packed + (size_t)o * p.row_bytes;
  const bool b3 = p.format == QTEA_FMT_BASE3;
  const int per = b3 ? 5 : 4, bytes = b3 ? 26 : 32;
  const int lane_cols = per * lane;
  const bool lane_in = lane < bytes;
#pragma unroll 4
  for (int blk = 0; blk < n_blocks; ++blk) {
    const int g = (blk * 128) / p.group_size;
    const uint16_t* sc = p.scales + ((size_t)o * p.G + g) * (p.bias ? 2 : 1);
    const float al = h2f(__ldg(sc)), be = p.bias ? h2f(__ldg(sc + 1)) : 0.f;
    const int c0 = blk * 128 + lane_cols;
    const bool on = lane_in && c0 < p.K && blk * bytes + lane < p.row_bytes;
    const uint32_t byte = on ? (uint32_t)__ldg(row + (size_t)blk * bytes + lane) : 0x55u;
    const uint32_t codes = b3 ? (uint32_t)lut[min(byte, 242u)] : byte;  // 2-bit codes, lowest column first
    float tvx[MB], sx[MB];
#pragma unroll
    for (int m = 0; m < MB; ++m) tvx[m] = sx[m] = 0.f;
#pragma unroll
    for (int d = 0; d < 5; ++d) {
      const int col = c0 + d;
      const bool cin = on && d < per && col < p.K && lane_cols + d < 128;
      const int t = (int)((codes >> (2 * d)) & 3u) - 1;
      const float vj = cin ? h2f(__ldg(p.v + col)) : 0.f;
#pragma unroll
      for (int m = 0; m < MB; ++m) {
        if (m < M) {
          const float xj = cin ? h2f(__ldg(p.x + (size_t)m * p.K + col)) : 0.f;
          sx[m] += xj;
          const float xv = vj * xj;  // exact in fp32
          tvx[m] += t > 0 ? xv : (t < 0 ? -xv : 0.f);
        }
      }
    }
#pragma unroll
    for (int m = 0; m < MB; ++m) acc[m] += al * tvx[m] + be * sx[m];
  }
  if (p.s > 0) {
    // lane takes entries lane, lane + 32, ...; four at a time, with the position bytes, salient
    // columns and values of all four loaded before any is used, then their x
    const int q = o >> 2, pos = o & 3, rs = (p.s + 3) / 4;
    for (int c0 = lane; c0 < p.s; c0 += 128) {
      uint32_t pb[4];
      int jj[4];
      float r[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int c = c0 + 32 * k;
        const bool in = c < p.s;
        pb[k] = in ? __ldg(p.ridx + (size_t)q * rs + (c >> 2)) : 0u;
        jj[k] = in ? __ldg(p.sal + c) : 0;
        const size_t e = (size_t)q * p.s + c;
        r[k] = !in ? 0.f
                   : p.residual_fp8 ? e4m3_to_float(__ldg(reinterpret_cast<const uint8_t*>(p.rvals) + e))
                                    : h2f(__ldg(reinterpret_cast<const uint16_t*>(p.rvals) + e));
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int c = c0 + 32 * k;
        if (c >= p.s || ((pb[k] >> (2 * (c & 3))) & 3u) != (uint32_t)pos) continue;
        const int j = jj[k] < 0 ? 0 : (jj[k] >= p.K ? p.K - 1 : jj[k]);
#pragma unroll
        for (int m = 0; m < MB; ++m)
          if (m < M) res[m] += r[k] * h2f(__ldg(p.x + (size_t)m * p.K + j));
      }
    }
  }
#pragma unroll
  for (int m = 0; m < MB; ++m) {
    float a = acc[m], r = res[m];
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      a += __shfl_xor_sync(0xffffffffu, a, off);
      r += __shfl_xor_sync(0xffffffffu, r, off);
    }
    if (lane == 0 && m < M) p.y[(size_t)m * p.N + o] = a + r;
  }
}

// The same product with the activations staged once per CTA (M <= 4, when v*x of every batch row,
// the per-group sums of x and the base-3 table fit in shared memory): each CTA writes
// x~[m][j] = v_j * x[m][j] (exact in fp32) and, with beta, sum_{j in g} x[m][j] (partial sums of
// eight columns, then a fixed order), then its warps walk rows. A warp loads 26 code bytes per
// lane (832 consecutive bytes of the row) before decoding any; lane l takes bytes l, l + 32, ...,
// so the columns of a load instruction are 4 or 5 apart and their x~ lie in distinct banks. Each
// byte adds alpha_g * sum T x~ over its columns; beta * sum x is added once per group.
constexpr int kStagedWarps = 16;
constexpr int kStagedBatch = 26;

size_t staged_smem_bytes(int M, int K, int G, bool bias) {
  return (size_t)M * K * sizeof(float) + (bias ? (size_t)M * G * sizeof(float) : 0) +
         (size_t)M * ((K + 7) / 8) * sizeof(float) + 256 * sizeof(uint16_t);
}

template <int MB, bool B3>
__global__ void __launch_bounds__(kStagedWarps * 32) qtea_gemv_paper_staged_kernel(const PaperParams p) {
  extern __shared__ __align__(16) float smf[];
  const int K = p.K, G = p.G, M = p.M;
  const int K8 = (K + 7) / 8;
  float* xt = smf;                                     // [M][K]
  float* sx = xt + (size_t)M * K;                      // [M][G], with beta
  float* s8 = sx + (p.bias ? (size_t)M * G : 0);       // [M][K8] sums of x over eight columns
  uint16_t* lut = reinterpret_cast<uint16_t*>(s8 + (size_t)M * K8);  // [243]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (B3)
    for (int i = threadIdx.x; i < 243; i += blockDim.x) {
      int b = i;
      uint32_t v = 0;
      for (int d = 0; d < 5; ++d) {
        v |= (uint32_t)(b % 3) << (2 * d);
        b /= 3;
      }
      lut[i] = (uint16_t)v;
    }
  // x~ and eight-column sums of x: 16-byte loads where x and v are 16-byte aligned and K % 8 == 0
  const bool vec = (K & 7) == 0 && ((reinterpret_cast<uintptr_t>(p.x) | reinterpret_cast<uintptr_t>(p.v)) & 15) == 0;
  if (vec) {
    constexpr int kU = 4;
    for (int t0 = threadIdx.x; t0 < M * K8; t0 += kU * blockDim.x) {
      uint4 xv[kU], vv[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int t = t0 + u * blockDim.x;
        if (t < M * K8) {
          const int m = t / K8, j8 = t - m * K8;
          xv[u] = __ldg(reinterpret_cast<const uint4*>(p.x + (size_t)m * K) + j8);
          vv[u] = __ldg(reinterpret_cast<const uint4*>(p.v) + j8);
        }
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int t = t0 + u * blockDim.x;
        if (t >= M * K8) continue;
        const int m = t / K8, j8 = t - m * K8;
        const uint32_t xw[4] = {xv[u].x, xv[u].y, xv[u].z, xv[u].w}, vw[4] = {vv[u].x, vv[u].y, vv[u].z, vv[u].w};
        float sum8 = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float xe = h2f((uint16_t)(xw[e >> 1] >> (16 * (e & 1))));
          const float ve = h2f((uint16_t)(vw[e >> 1] >> (16 * (e & 1))));
          xt[(size_t)m * K + 8 * j8 + e] = ve * xe;
          sum8 += xe;
        }
        s8[t] = sum8;
      }
    }
  } else {
    for (int t = threadIdx.x; t < M * K8; t += blockDim.x) {
      const int m = t / K8, j8 = t - m * K8;
      float sum8 = 0.f;
      for (int e = 0; e < 8; ++e) {
        const int j = 8 * j8 + e;
        if (j >= K) break;
        const float xe = h2f(__ldg(p.x + (size_t)m * K + j));
        xt[(size_t)m * K + j] = h2f(__ldg(p.v + j)) * xe;
        sum8 += xe;
      }
      s8[t] = sum8;
    }
  }
  __syncthreads();
  if (p.bias)  // groups are K or 128 columns: whole eight-column blocks, summed in order
    for (int t = threadIdx.x; t < M * G; t += blockDim.x) {
      const int m = t / G, g = t - m * G;
      const int b0 = g * p.group_size / 8, b1 = min(K8, (g * p.group_size + p.group_size + 7) / 8);
      float a = 0.f;
      for (int b8 = b0; b8 < b1; ++b8) a += s8[(size_t)m * K8 + b8];
      sx[t] = a;
    }
  __syncthreads();

  const int per = B3 ? 5 : 4, bytes = B3 ? 26 : 32;
  const int sc_stride = p.bias ? 2 : 1;
  for (int o = blockIdx.x * kStagedWarps + warp; o < p.N; o += gridDim.x * kStagedWarps) {
    const uint8_t* row = p.packed + (size_t)o * p.row_bytes;
    const uint16_t* sc = p.scales + (size_t)o * G * sc_stride;
    // bring the row's scales into L1 ahead of the per-byte lookups
    float warm = 0.f;
    for (int e = 2 * lane; e < G * sc_stride; e += 64) warm += h2f(__ldg(sc + e));
    float acc[MB];
#pragma unroll
    for (int m = 0; m < MB; ++m) acc[m] = 0.f;
    for (int i0 = 0; i0 < p.row_bytes; i0 += 32 * kStagedBatch) {
      uint32_t byte[kStagedBatch];
#pragma unroll
      for (int k = 0; k < kStagedBatch; ++k) {
        const int i = i0 + lane + 32 * k;
        byte[k] = i < p.row_bytes ? (uint32_t)__ldg(row + i) : 0xFFFFFFFFu;
      }
#pragma unroll
      for (int k = 0; k < kStagedBatch; ++k) {
        if (byte[k] == 0xFFFFFFFFu) continue;
        const int i = i0 + lane + 32 * k;
        const int blk = i / bytes, q = i - blk * bytes;
        const int c0 = blk * 128 + per * q;
        if (c0 >= K) continue;
        const float al = h2f(__ldg(sc + (size_t)((blk * 128) / p.group_size) * sc_stride));
        const uint32_t codes = B3 ? (uint32_t)lut[min(byte[k], 242u)] : byte[k];
        float part[MB];
#pragma unroll
        for (int m = 0; m < MB; ++m) part[m] = 0.f;
#pragma unroll
        for (int d = 0; d < per; ++d) {
          const int col = c0 + d;
          if ((B3 && per * q + d >= 128) || col >= K) continue;
          const uint32_t c = (codes >> (2 * d)) & 3u;
#pragma unroll
          for (int m = 0; m < MB; ++m) {
            if (m < M) {
              const float xv = xt[(size_t)m * K + col];
              part[m] += c == 2u ? xv : (c == 0u ? -xv : 0.f);
            }
          }
        }
#pragma unroll
        for (int m = 0; m < MB; ++m) acc[m] += al * part[m];
      }
    }
    acc[0] += warm * 0.f;  // keeps the warming loads (adds zero)
    if (p.bias)
      for (int g = lane; g < G; g += 32) {
        const float be = h2f(__ldg(sc + (size_t)g * 2 + 1));
#pragma unroll
        for (int m = 0; m < MB; ++m)
          if (m < M) acc[m] += be * sx[(size_t)m * G + g];
      }
    float res[MB];
#pragma unroll
    for (int m = 0; m < MB; ++m) res[m] = 0.f;
    if (p.s > 0) {
      const int q4 = o >> 2, pos = o & 3, rs = (p.s + 3) / 4;
      for (int c0 = lane; c0 < p.s; c0 += 128) {
        uint32_t pb[4];
        int jj[4];
        float r[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int c = c0 + 32 * k;
          const bool in = c < p.s;
          pb[k] = in ? __ldg(p.ridx + (size_t)q4 * rs + (c >> 2)) : 0u;
          jj[k] = in ? __ldg(p.sal + c) : 0;
          const size_t e = (size_t)q4 * p.s + c;
          r[k] = !in ? 0.f
                     : p.residual_fp8 ? e4m3_to_float(__ldg(reinterpret_cast<const uint8_t*>(p.rvals) + e))
                                      : h2f(__ldg(reinterpret_cast<const uint16_t*>(p.rvals) + e));
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int c = c0 + 32 * k;
          if (c >= p.s || ((pb[k] >> (2 * (c & 3))) & 3u) != (uint32_t)pos) continue;
          const int j = jj[k] < 0 ? 0 : (jj[k] >= K ? K - 1 : jj[k]);
#pragma unroll
          for (int m = 0; m < MB; ++m)
            if (m < M) res[m] += r[k] * h2f(__ldg(p.x + (size_t)m * K + j));
        }
      }
    }
#pragma unroll
    for (int m = 0; m < MB; ++m) {
      float a = acc[m], r = res[m];
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, off);
        r += __shfl_xor_sync(0xffffffffu, r, off);
      }
      if (lane == 0 && m < M) p.y[(size_t)m * p.N + o] = a + r;
    }
  }
}

// Base-3 layouts with staged activations in fixed point (M <= 4): per batch row and 128-column block
// the CTA scales x~ = v*x by a power of two so that |X| < 2^22 (X = round(x~ * 2^e), e from the
// block's largest |x~|) and splits X into three byte planes (low and middle unsigned, top signed).
// The block's 26 code bytes are taken four at a time (seven groups, the last two bytes of the
// seventh standing for columns past the block, X = 0 there). Per group one 64-byte record: for each
// plane, the four bytes' first four columns (one word per byte), then the four bytes' fifth
// columns in one word per plane, and S = sum of the group's X. A 243-entry table turns a code byte
// into a word of its first four codes c = T + 1 and its fifth code. Per group, sum c X is fifteen
// dp4a, exact in int32; sum T X = that - S, summed over the block and scaled once by alpha * 2^-e.
// Outliers: values of x~ at least 16 times above the rest of the block (found in rounds, as in the
// batch-1 kernel) are taken out of the planes, up to kB3MaxOut per block, and added exactly in fp32:
// T x~ with T read from the row's code byte. The rest set the scale: |X| < 2^23.
// The rounding of X is the only approximation: |x~ - X 2^-e| <= 2^-e / 2 with
// 2^-e <= 2^-22 * max|x~| over the block's values that are not outliers.
constexpr int kB3Groups = 7;        // groups of four code bytes per block
constexpr int kB3GroupWords = 16;   // words per group record
constexpr int kB3BlockWords = 116;  // 7 x 16 words plus 4 (outliers: count and columns, then up to
                                    // three values); lanes that read different blocks' records hit
                                    // distinct banks
constexpr int kB3MaxOut = 3;

// Shared memory of one base-3 problem after the 256-entry table: records, 2^-e and block sums of x
// per batch row and block, and the per-group sums of x with beta.
size_t b3_region_bytes(int M, int K, int G, bool bias) {
  const size_t n_blocks = (size_t)(K + 127) / 128;
  return (size_t)M * n_blocks * kB3BlockWords * sizeof(uint32_t) + 2 * (size_t)M * n_blocks * sizeof(float) +
         (bias ? (size_t)M * G * sizeof(float) : 0);
}

template <int MB>
__device__ void b3_problem(const PaperParams& p, int row_lo, int row_hi, uint32_t* smw, const uint2* lut) {
  const int K = p.K, G = p.G, M = p.M;
  const int n_blocks = (K + 127) / 128;
  uint32_t* rec = smw;                                                    // [M][n_blocks][212]
  float* inv = reinterpret_cast<float*>(rec + (size_t)M * n_blocks * kB3BlockWords);  // [M][n_blocks] 2^-e
  float* sx = inv + (size_t)M * n_blocks;                                 // [M][G] sum of x, with beta
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // one warp per (batch row, block), two tasks' loads in flight: lane q < 26 owns columns
  // 5q .. 5q+4 of the block; the warp also sums the block's x for the beta term
  float* bx = sx + (p.bias ? (size_t)M * G : 0);  // [M][n_blocks], in the slack before the table
  for (int t0 = warp; t0 < M * n_blocks; t0 += 2 * kStagedWarps) {
    float xv[2][5], vv[2][5];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int t = t0 + u * kStagedWarps;
      const int m = t / n_blocks, blk = t - m * n_blocks;
#pragma unroll
      for (int d = 0; d < 5; ++d) {
        const int cb = 5 * lane + d, col = blk * 128 + cb;
        const bool in = t < M * n_blocks && lane < 26 && cb < 128 && col < K;
        xv[u][d] = in ? h2f(__ldg(p.x + (size_t)m * K + col)) : 0.f;
        vv[u][d] = in ? h2f(__ldg(p.v + col)) : 0.f;
      }
    }
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int t = t0 + u * kStagedWarps;
      if (t >= M * n_blocks) break;  // warp-uniform
      float xt[5];
      float amax = 0.f, xs = 0.f;
#pragma unroll
      for (int d = 0; d < 5; ++d) {
        xt[d] = vv[u][d] * xv[u][d];
        amax = fmaxf(amax, fabsf(xt[d]));
        xs += xv[u][d];
      }
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
        xs += __shfl_xor_sync(0xffffffffu, xs, off);
      }
      uint32_t outm = 0;  // bit d: xt[d] is an outlier
      int n_out = 0;
#pragma unroll 1
      for (int round = 0; round < kB3MaxOut && amax > 0.f; ++round) {
        const float thr = amax * 0.0625f;
        uint32_t m = 0;
#pragma unroll
        for (int d = 0; d < 5; ++d) m |= (fabsf(xt[d]) > thr ? 1u : 0u) << d;
        m &= ~outm;
        const int c = (int)__reduce_add_sync(0xffffffffu, (unsigned)__popc(m));
        if (c > kB3MaxOut - n_out) break;
        outm |= m;
        n_out += c;
        float lm = 0.f;
#pragma unroll
        for (int d = 0; d < 5; ++d) lm = fmaxf(lm, ((outm >> d) & 1u) ? 0.f : fabsf(xt[d]));
#pragma unroll
        for (int off = 16; off; off >>= 1) lm = fmaxf(lm, __shfl_xor_sync(0xffffffffu, lm, off));
        amax = lm;
      }
      int ex = 0;
      if (amax > 0.f) frexpf(amax, &ex);  // amax < 2^ex
      const int e = 23 - ex;              // |X| <= 2^23 * amax / 2^ex: at most 2^23 - 1 after the clamp
      // lane q owns code byte q of the block (columns 5q .. 5q+4; lanes 26 and 27 stand for the two
      // padding bytes of the seventh group and hold X = 0)
      uint32_t a0 = 0, a1 = 0, a2 = 0, f0 = 0, f1 = 0, f2 = 0;
      int sum = 0;
#pragma unroll
      for (int d = 0; d < 5; ++d) {
        const int X = (amax > 0.f && !((outm >> d) & 1u)) ? min(__float2int_rn(ldexpf(xt[d], e)), 8388607) : 0;
        sum += X;
        const uint32_t u0 = (uint32_t)X & 0xFFu, u1 = ((uint32_t)X >> 8) & 0xFFu, u2 = ((uint32_t)X >> 16) & 0xFFu;
        if (d < 4) {
          a0 |= u0 << (8 * d);
          a1 |= u1 << (8 * d);
          a2 |= u2 << (8 * d);
        } else {
          f0 = u0;
          f1 = u1;
          f2 = u2;
        }
      }
      // the group's fifth columns, byte i from lane 4 (q / 4) + i, and the group's sum of X
      uint32_t w0 = 0, w1 = 0, w2 = 0;
      int gsum = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int src = (lane & ~3) + i;
        w0 |= __shfl_sync(0xffffffffu, f0, src) << (8 * i);
        w1 |= __shfl_sync(0xffffffffu, f1, src) << (8 * i);
        w2 |= __shfl_sync(0xffffffffu, f2, src) << (8 * i);
        gsum += __shfl_sync(0xffffffffu, sum, src);
      }
      if (lane < 4 * kB3Groups) {
        uint32_t* r = rec + (size_t)t * kB3BlockWords + (lane >> 2) * kB3GroupWords;
        const int b = lane & 3;
        r[b] = a0;
        r[4 + b] = a1;
        r[8 + b] = a2;
        if (b == 0) *reinterpret_cast<uint4*>(r + 12) = make_uint4(w0, w1, w2, (uint32_t)gsum);
      }
      {  // the outlier list in the record's last four words: count and columns, then the values
        uint32_t* ol = rec + (size_t)t * kB3BlockWords + kB3Groups * kB3GroupWords;
        const int mine = __popc(outm);
        int off = mine;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(0xffffffffu, off, o);
          if (lane >= o) off += v;
        }
        off -= mine;  // earlier lanes' outliers
        uint32_t cols = 0;
#pragma unroll
        for (int d = 0; d < 5; ++d)
          if ((outm >> d) & 1u) {
            ol[1 + off] = __float_as_uint(xt[d]);
            cols |= (uint32_t)(5 * lane + d) << (8 * (1 + off));
            ++off;
          }
        cols = __reduce_or_sync(0xffffffffu, cols);
        if (lane == 0) ol[0] = cols | (uint32_t)n_out;
      }
      if (lane == 0) {
        inv[t] = amax > 0.f ? ldexpf(1.f, -e) : 0.f;
        bx[t] = xs;
      }
    }
  }
  __syncthreads();
  if (p.bias)  // groups of 128 columns are the blocks; a whole-row group sums the blocks in order
    for (int t = threadIdx.x; t < M * G; t += blockDim.x) {
      const int m = t / G, g = t - m * G;
      float a = 0.f;
      if (p.group_size >= K)
        for (int blk = 0; blk < n_blocks; ++blk) a += bx[m * n_blocks + blk];
      else
        a = bx[m * n_blocks + g];
      sx[t] = a;
    }
  __syncthreads();

  const bool row_group = p.group_size >= K;  // one scale group per row
  const int sc_stride = p.bias ? 2 : 1;
  for (int o = row_lo + warp; o < row_hi; o += kStagedWarps) {
    const uint8_t* row = p.packed + (size_t)o * p.row_bytes;
    const uint16_t* sc = p.scales + (size_t)o * G * sc_stride;
    float acc[MB];
#pragma unroll
    for (int m = 0; m < MB; ++m) acc[m] = 0.f;
    // lane l takes block b0 + l of the row: its 26 code bytes (13 two-byte loads), one alpha, and
    // an int32 sum over the block (|sum_j T_j X_j| < 128 * 2^22), converted once
    for (int b0 = 0; b0 < n_blocks; b0 += 32) {
      const int blk = b0 + lane;
      const bool on = blk < n_blocks;
      const uint16_t* cb = reinterpret_cast<const uint16_t*>(row + (size_t)(on ? blk : 0) * 26);
      uint32_t h[13];
#pragma unroll
      for (int k = 0; k < 13; ++k) h[k] = on ? (uint32_t)__ldg(cb + k) : 0x7979u;  // 121 = five T = 0 digits
      const float al = on ? h2f(__ldg(sc + (row_group ? 0 : (size_t)blk * sc_stride))) : 0.f;
      int isum[MB];
#pragma unroll
      for (int m = 0; m < MB; ++m) isum[m] = 0;
#pragma unroll
      for (int gq = 0; gq < kB3Groups; ++gq) {
        uint2 cw[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int j = 4 * gq + i;  // bytes 26 and 27 stand for columns past the block: T = 0
          const uint32_t byte = j < 26 ? (h[j >> 1] >> (8 * (j & 1))) & 0xFFu : 121u;
          cw[i] = lut[byte];
        }
        const uint32_t c4 = cw[0].y | (cw[1].y << 8) | (cw[2].y << 16) | (cw[3].y << 24);
#pragma unroll
        for (int m = 0; m < MB; ++m) {
          if (m < M) {
            const uint4* r = reinterpret_cast<const uint4*>(
                rec + (size_t)(m * n_blocks + (on ? blk : 0)) * kB3BlockWords + gq * kB3GroupWords);
            const uint4 p0 = r[0], p1 = r[1], p2 = r[2], ft = r[3];
            int s0 = __dp4a(cw[0].x, p0.x, __dp4a(cw[1].x, p0.y, __dp4a(cw[2].x, p0.z, __dp4a(cw[3].x, p0.w, 0u))));
            int s1 = __dp4a(cw[0].x, p1.x, __dp4a(cw[1].x, p1.y, __dp4a(cw[2].x, p1.z, __dp4a(cw[3].x, p1.w, 0u))));
            int s2 = __dp4a((int)cw[0].x, (int)p2.x,
                            __dp4a((int)cw[1].x, (int)p2.y, __dp4a((int)cw[2].x, (int)p2.z, __dp4a((int)cw[3].x, (int)p2.w, 0))));
            s0 = __dp4a(c4, ft.x, (unsigned)s0);
            s1 = __dp4a(c4, ft.y, (unsigned)s1);
            s2 = __dp4a((int)c4, (int)ft.z, s2);
            isum[m] += s2 * 65536 + s1 * 256 + s0 - (int)ft.w;
          }
        }
      }
      if (on)
#pragma unroll
        for (int m = 0; m < MB; ++m)
          if (m < M) {
            // the block's outliers: T x~ in fp32, T from the code byte (reloaded: a register array
            // indexed by a loop value would go to local memory)
            const uint32_t* ol = rec + (size_t)(m * n_blocks + blk) * kB3BlockWords + kB3Groups * kB3GroupWords;
            const uint32_t head = ol[0];
            float ov = 0.f;
            for (int k = 0; k < (int)(head & 0xFFu); ++k) {
              const int c = (int)((head >> (8 * (1 + k))) & 0xFFu);
              const uint2 cw = lut[__ldg(row + (size_t)blk * 26 + c / 5)];
              const int d = c % 5;
              const int code = d < 4 ? (int)((cw.x >> (8 * d)) & 0xFFu) : (int)cw.y;
              ov = fmaf((float)(code - 1), __uint_as_float(ol[1 + k]), ov);
            }
            acc[m] += al * fmaf(inv[m * n_blocks + blk], (float)isum[m], ov);
          }
    }
    if (p.bias)
      for (int g = lane; g < G; g += 32) {
        const float be = h2f(__ldg(sc + (size_t)g * 2 + 1));
#pragma unroll
        for (int m = 0; m < MB; ++m)
          if (m < M) acc[m] += be * sx[(size_t)m * G + g];
      }
    float res[MB];
#pragma unroll
    for (int m = 0; m < MB; ++m) res[m] = 0.f;
    if (p.s > 0) {
      const int q4 = o >> 2, pos = o & 3, rs = (p.s + 3) / 4;
      for (int c0 = lane; c0 < p.s; c0 += 128) {
        uint32_t pb[4];
        int jj[4];
        float r[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int c = c0 + 32 * k;
          const bool in = c < p.s;
          pb[k] = in ? __ldg(p.ridx + (size_t)q4 * rs + (c >> 2)) : 0u;
          jj[k] = in ? __ldg(p.sal + c) : 0;
          const size_t e = (size_t)q4 * p.s + c;
          r[k] = !in ? 0.f
                     : p.residual_fp8 ? e4m3_to_float(__ldg(reinterpret_cast<const uint8_t*>(p.rvals) + e))
                                      : h2f(__ldg(reinterpret_cast<const uint16_t*>(p.rvals) + e));
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int c = c0 + 32 * k;
          if (c >= p.s || ((pb[k] >> (2 * (c & 3))) & 3u) != (uint32_t)pos) continue;
          const int j = jj[k] < 0 ? 0 : (jj[k] >= K ? K - 1 : jj[k]);
#pragma unroll
          for (int m = 0; m < MB; ++m)
            if (m < M) res[m] += r[k] * h2f(__ldg(p.x + (size_t)m * K + j));
        }
      }
    }
#pragma unroll
    for (int m = 0; m < MB; ++m) {
      float a = acc[m], r = res[m];
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, off);
        r += __shfl_xor_sync(0xffffffffu, r, off);
      }
      if (lane == 0 && m < M) p.y[(size_t)m * p.N + o] = a + r;
    }
  }
}

// The base-3 problems of a grouped call in one launch. The rows of all problems, each weighted by
// its blocks, are split evenly over the persistent CTAs; a CTA stages a problem once for the rows
// of it that fall in its share (one or two problems for most CTAs).
template <int MB>
__global__ void __launch_bounds__(kStagedWarps * 32) qtea_gemv_paper_b3_kernel(const B3Group g) {
  extern __shared__ __align__(16) uint32_t smw[];
  uint2* lut = reinterpret_cast<uint2*>(smw);  // [256]
  for (int i = threadIdx.x; i < 256; i += blockDim.x) {  // bytes above 242 never occur; T = 0 there
    int b = i < 243 ? i : 121;
    uint32_t w1 = 0, w2 = 0;
    for (int d = 0; d < 5; ++d) {
      const uint32_t c = (uint32_t)(b % 3);
      b /= 3;
      if (d < 4) w1 |= c << (8 * d);
      else w2 = c;
    }
    lut[i] = make_uint2(w1, w2);
  }
  const long long total = g.work[g.n];
  const long long lo = total * blockIdx.x / gridDim.x, hi = total * (blockIdx.x + 1) / gridDim.x;
  for (int q = 0; q < g.n; ++q) {
    const long long w0 = g.work[q], w1 = g.work[q + 1];
    const long long a = lo > w0 ? lo : w0, b = hi < w1 ? hi : w1;
    if (a >= b) continue;
    const int nb = (g.prob[q].K + 127) / 128;
    // row r belongs to the CTA whose share holds its first block
    const int row_lo = (int)((a - w0 + nb - 1) / nb), row_hi = (int)((b - w0 + nb - 1) / nb);
    if (row_lo >= row_hi) continue;
    __syncthreads();  // the previous problem's rows are done with the staged data
    b3_problem<MB>(g.prob[q], row_lo, row_hi, smw + 512, lut);
  }
}

// Base-3 packing (Sec. 3.5): per row, K_pad3 / 128 groups of 26 bytes; byte q of a group holds
// columns 5q .. 5q+4 of the group as sum_d (T + 1) 3^d, the lowest column in the least significant
// digit. Byte 25 holds columns 125-127 and two pad digits; pad digits and columns >= K are digit 1
// (T = 0). One thread per byte; any code outside {-1, 0, +1} sets *bad_flag.
__global__ void qtea_pack_base3_kernel(const int8_t* __restrict__ codes, int N, int K, int groups,
                                       uint8_t* __restrict__ packed, int* bad_flag) {
  const long long n_bytes = (long long)N * groups * 26;
  bool bad = false;
  for (long long bi = blockIdx.x * (long long)blockDim.x + threadIdx.x; bi < n_bytes;
       bi += (long long)gridDim.x * blockDim.x) {
    const long long r = bi / ((long long)groups * 26);
    const int rem = (int)(bi - r * groups * 26);
    const int h = rem / 26, q = rem - h * 26;
    int value = 0, weight = 1;
    for (int d = 0; d < 5; ++d) {
      const int in_group = 5 * q + d;
      const int col = 128 * h + in_group;
      int digit = 1;
      if (in_group < 128 && col < K) {
        const int t = codes[r * (long long)K + col];
        bad |= (t < -1 || t > 1);
        digit = t + 1;
      }
      value += digit * weight;
      weight *= 3;
    }
    packed[bi] = (uint8_t)value;
  }
  if (bad) atomicExch(bad_flag, 1);
}

}  // namespace

template <int MB, bool B3>
cudaError_t launch_staged(const PaperParams& p, size_t smem, cudaStream_t st) {
  int per_sm = 1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, qtea_gemv_paper_staged_kernel<MB, B3>, kStagedWarps * 32,
                                                    smem) != cudaSuccess)
    return cudaGetLastError();
  const int want = (p.N + kStagedWarps - 1) / kStagedWarps;
  const int grid = std::max(1, std::min(want, p.sm_count * std::max(per_sm, 1)));
  qtea_gemv_paper_staged_kernel<MB, B3><<<grid, kStagedWarps * 32, smem, st>>>(p);
  return cudaGetLastError();
}

template <int MB>
cudaError_t launch_b3_group(const B3Group& g, size_t smem, int sm_count, cudaStream_t st) {
  int per_sm = 1;  // resident CTAs per SM: the grid is persistent, so each CTA stages once per problem
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, qtea_gemv_paper_b3_kernel<MB>, kStagedWarps * 32, smem) !=
      cudaSuccess)
    return cudaGetLastError();
  long long rows = 0;
  for (int q = 0; q < g.n; ++q) rows += g.prob[q].N;
  const long long want = (rows + kStagedWarps - 1) / kStagedWarps;
  const int grid = (int)std::max<long long>(1, std::min<long long>(want, (long long)sm_count * std::max(per_sm, 1)));
  qtea_gemv_paper_b3_kernel<MB><<<grid, kStagedWarps * 32, smem, st>>>(g);
  return cudaGetLastError();
}

size_t b3_smem_bytes(int M, int K, int G, bool bias) { return 2048 + b3_region_bytes(M, K, G, bias) + 16; }

cudaError_t launch_b3(const B3Group& g, cudaStream_t st) {
  size_t smem = 0;
  for (int q = 0; q < g.n; ++q) {
    const PaperParams& p = g.prob[q];
    smem = std::max(smem, b3_smem_bytes(p.M, p.K, p.G, p.bias != 0));
  }
  const int M = g.n > 0 ? g.prob[0].M : 1, sm = g.n > 0 ? g.prob[0].sm_count : 1;
  if (M <= 1) return launch_b3_group<1>(g, smem, sm, st);
  if (M <= 2) return launch_b3_group<2>(g, smem, sm, st);
  return launch_b3_group<4>(g, smem, sm, st);
}

bool b3_eligible(const PaperParams& p) {
  return p.staged_ok && p.format == QTEA_FMT_BASE3 && p.M >= 1 && p.M <= 4 &&
         b3_smem_bytes(p.M, p.K, p.G, p.bias != 0) <= p.smem_optin;
}

cudaError_t paper_configure(size_t smem_optin) {
  const int dyn = (int)smem_optin;
  cudaError_t e;
#define QTEA_STAGED_ATTR(MB, B3)                                                                              \
  if ((e = cudaFuncSetAttribute(qtea_gemv_paper_staged_kernel<MB, B3>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                dyn)) != cudaSuccess)                                                          \
    return e;
  if ((e = cudaFuncSetAttribute(qtea_gemv_paper_b3_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn)) !=
      cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(qtea_gemv_paper_b3_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn)) !=
      cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(qtea_gemv_paper_b3_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn)) !=
      cudaSuccess)
    return e;
  QTEA_STAGED_ATTR(1, false)
  QTEA_STAGED_ATTR(2, false)
  QTEA_STAGED_ATTR(4, false)
#undef QTEA_STAGED_ATTR
  return cudaSuccess;
}

cudaError_t launch_paper(const PaperParams& p, cudaStream_t st) {
  const int grid = (p.N + kPaperWarps - 1) / kPaperWarps;
  if (grid == 0) return cudaSuccess;
  if (b3_eligible(p)) {
    B3Group g;
    g.prob[0] = p;
    g.n = 1;
    g.work[0] = 0;
    g.work[1] = (long long)p.N * ((p.K + 127) / 128);
    return launch_b3(g, st);
  }
  const size_t smem = staged_smem_bytes(p.M, p.K, p.G, p.bias != 0);
  if (p.staged_ok && p.M <= 4 && p.format != QTEA_FMT_BASE3 && smem <= p.smem_optin) {
    if (p.M <= 1) return launch_staged<1, false>(p, smem, st);
    if (p.M <= 2) return launch_staged<2, false>(p, smem, st);
    return launch_staged<4, false>(p, smem, st);
  }
  const int threads = kPaperWarps * 32;
  if (p.M <= 1) qtea_gemv_paper_kernel<1><<<grid, threads, 0, st>>>(p);
  else if (p.M <= 2) qtea_gemv_paper_kernel<2><<<grid, threads, 0, st>>>(p);
  else if (p.M <= 4) qtea_gemv_paper_kernel<4><<<grid, threads, 0, st>>>(p);
  else if (p.M <= 8) qtea_gemv_paper_kernel<8><<<grid, threads, 0, st>>>(p);
  else qtea_gemv_paper_kernel<16><<<grid, threads, 0, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_pack_base3(const int8_t* codes, int N, int K, uint8_t* packed, int* bad_flag, cudaStream_t st) {
  const int groups = (K + 127) / 128;
  const long long n_bytes = (long long)N * groups * 26;
  if (n_bytes == 0) return cudaSuccess;
  const int threads = 256;
  long long blocks = (n_bytes + threads - 1) / threads;
  if (blocks > 65536) blocks = 65536;
  qtea_pack_base3_kernel<<<(int)blocks, threads, 0, st>>>(codes, N, K, groups, packed, bad_flag);
  return cudaGetLastError();
}

}  // namespace qtea
