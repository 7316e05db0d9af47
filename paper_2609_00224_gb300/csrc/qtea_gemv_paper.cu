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
// One warp per output row. Lane l takes the row's 128-column blocks l, l + 32, ...; a block lies in
// one scale group (groups are 128 columns or the whole row), so the lane adds
// alpha * sum T v x + beta * sum x once per block and batch row. Base-3 bytes are expanded to five
// 2-bit codes through a 243-entry table in shared memory. v*x is exact in fp32; sums are fp32.
// The same warp adds the residual of the row's group of four.
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

// Codes (T + 1, 2 bits each, lowest column first) of the 128-column block `blk` of row `row`:
// 8 words. Columns at or beyond K hold code 1.
__device__ __forceinline__ void block_codes(const PaperParams& p, int row, int blk, const uint16_t* lut,
                                            uint32_t (&w)[8]) {
  if (p.format == QTEA_FMT_2BIT) {
    // rows are K_pad/4 bytes, K_pad a multiple of 64: the last block may have only 64 columns
    const uint4* src = reinterpret_cast<const uint4*>(p.packed + (size_t)row * p.row_bytes + (size_t)blk * 32);
    const uint4 a = __ldg(src);
    const uint4 b = blk * 32 + 16 < p.row_bytes ? __ldg(src + 1) : make_uint4(0x55555555u, 0x55555555u, 0x55555555u,
                                                                              0x55555555u);
    w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
    w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
  } else {
    // 26 bytes: byte q holds columns 5q .. 5q+4 as base-3 digits; byte 25 covers columns 125-127
    const uint8_t* src = p.packed + (size_t)row * p.row_bytes + (size_t)blk * 26;
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = 0;
#pragma unroll
    for (int q = 0; q < 26; ++q) {
      const uint32_t c5 = lut[min((uint32_t)__ldg(src + q), 242u)];  // five 2-bit codes (bytes are < 243)
#pragma unroll
      for (int d = 0; d < 5; ++d) {
        const int col = 5 * q + d;
        if (col < 128) w[col >> 4] |= ((c5 >> (2 * d)) & 3u) << (2 * (col & 15));
      }
    }
  }
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

  const int n_blocks = (p.K + 127) / 128;
  for (int blk = lane; blk < n_blocks; blk += 32) {
    uint32_t w[8];
    block_codes(p, o, blk, lut, w);
    const int g = (blk * 128) / p.group_size;
    const uint16_t* sc = p.scales + ((size_t)o * p.G + g) * (p.bias ? 2 : 1);
    const float al = h2f(__ldg(sc)), be = p.bias ? h2f(__ldg(sc + 1)) : 0.f;
    float tvx[MB], sx[MB];
#pragma unroll
    for (int m = 0; m < MB; ++m) tvx[m] = sx[m] = 0.f;
    const int c0 = blk * 128;
    for (int i = 0; i < 128; ++i) {
      const int col = c0 + i;
      if (col >= p.K) break;
      const int t = (int)((w[i >> 4] >> (2 * (i & 15))) & 3u) - 1;
      const float vj = h2f(__ldg(p.v + col));
#pragma unroll
      for (int m = 0; m < MB; ++m) {
        if (m < M) {
          const float xj = h2f(__ldg(p.x + (size_t)m * p.K + col));
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
    const int q = o >> 2, pos = o & 3, rs = (p.s + 3) / 4;
    for (int c = lane; c < p.s; c += 32) {
      if (((p.ridx[(size_t)q * rs + (c >> 2)] >> (2 * (c & 3))) & 3) != pos) continue;
      int j = p.sal[c];
      j = j < 0 ? 0 : (j >= p.K ? p.K - 1 : j);
      const size_t e = (size_t)q * p.s + c;
      const float r = p.residual_fp8 ? e4m3_to_float(reinterpret_cast<const uint8_t*>(p.rvals)[e])
                                     : h2f(reinterpret_cast<const uint16_t*>(p.rvals)[e]);
#pragma unroll
      for (int m = 0; m < MB; ++m)
        if (m < M) res[m] += r * h2f(p.x[(size_t)m * p.K + j]);
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
