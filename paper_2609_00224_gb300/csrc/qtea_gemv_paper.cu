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
// One warp per output row, walking the row's 128-column blocks; a block lies in one scale group
// (groups are 128 columns or the whole row). Lane l takes code byte l of the block and adds
// alpha * sum T v x + beta * sum x over its columns for every batch row; the lanes' sums are added
// once at the end. Base-3 bytes are expanded to five 2-bit codes through a 243-entry table in shared
// memory. v*x is exact in fp32; sums are fp32. The same warp adds the residual of the row's group
// of four.
#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr int kPaperWarps = 4;

__device__ __forceinline__ float h2f(uint16_t b) { return __half2float(__ushort_as_half(b)); }

// FP8 E4M3 (sign bit 7, exponent bits 6-3 with bias 7, mantissa bits 2-0, subnormals at exponent
// 0, NaN at S.1111.111, no infinity) as fp32, exactly.
__device__ __forceinline__ float e4m3_to_float(uint32_t b) {
  const uint32_t e = (b >> 3) & 15u, m = b & 7u;
  float mag;
  if (e == 15u && m == 7u) {
    mag = __int_as_float(0x7fc00000);
  } else if (e == 0u) {
    mag = (float)m * 0.001953125f;  // m * 2^-9
  } else {
    mag = __int_as_float((int)((e + 120u) << 23 | m << 20));  // (1 + m/8) * 2^(e-7)
  }
  return (b & 0x80u) ? -mag : mag;
}

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

cudaError_t launch_paper(const PaperParams& p, cudaStream_t st) {
  const int grid = (p.N + kPaperWarps - 1) / kPaperWarps;
  if (grid == 0) return cudaSuccess;
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
