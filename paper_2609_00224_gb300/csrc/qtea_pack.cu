// Pack int8 ternary codes (Sec. 3.1, Eq. 2: T in {-1, 0, +1}) into the library's 2-bit layout:
// code T+1, four per byte, least significant first, rows padded to K_pad = K rounded up to a
// multiple of 64 with code 1. One thread writes one 32-bit word (16 codes). Any code outside
// {-1, 0, +1} sets *bad_flag; the packed bytes are then not used.
#include "qtea_internal.h"

namespace qtea {
namespace {

__global__ void qtea_pack_2bit_kernel(const int8_t* __restrict__ codes, int N, int K, int K_pad,
                                      uint32_t* __restrict__ packed, int* bad_flag) {
  const long long words_per_row = K_pad / 16;
  const long long n_words = (long long)N * words_per_row;
  bool bad = false;
  for (long long wi = blockIdx.x * (long long)blockDim.x + threadIdx.x; wi < n_words;
       wi += (long long)gridDim.x * blockDim.x) {
    const long long r = wi / words_per_row;
    const int col0 = (int)(wi % words_per_row) * 16;
    const int8_t* src = codes + r * (long long)K;
    uint32_t word = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int col = col0 + i;
      int code = 1;
      if (col < K) {
        const int t = src[col];
        bad |= (t < -1 || t > 1);
        code = t + 1;
      }
      word |= (uint32_t)(code & 3) << (2 * i);
    }
    packed[wi] = word;
  }
  if (bad) atomicExch(bad_flag, 1);
}

}  // namespace

cudaError_t launch_pack(const int8_t* codes, int N, int K, int K_pad, uint32_t* packed, int* bad_flag,
                        cudaStream_t st) {
  const long long n_words = (long long)N * (K_pad / 16);
  if (n_words == 0) return cudaSuccess;
  const int threads = 256;
  long long blocks = (n_words + threads - 1) / threads;
  if (blocks > 65536) blocks = 65536;
  qtea_pack_2bit_kernel<<<(int)blocks, threads, 0, st>>>(codes, N, K, K_pad, packed, bad_flag);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- salient bitmap (Sec. 3.5)
// The paper stores the salient set as a bitmap over the input columns (column j at bit j % 32 of
// word j / 32, least significant bit first); the GEMV takes the ascending index list.

constexpr int kBitmapThreads = 1024;

// The bitmap as the ascending index list, by one CTA: the words in tiles of kBitmapThreads, each
// word's population counted, scanned over its warp, and offset by the totals of the warps before
// it (every thread sums those itself from shared memory); each thread writes its word's columns at
// their rank. The first max_s indices are written, the count to *count.
__global__ void __launch_bounds__(kBitmapThreads) qtea_bitmap_to_index_kernel(const uint32_t* __restrict__ bitmap,
                                                                              int K, int32_t* __restrict__ idx,
                                                                              int max_s, int* count) {
  __shared__ int warp_tot[kBitmapThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_words = (K + 31) / 32;
  int base = 0;  // indices written by the earlier tiles (the same in every thread)
  for (int w0 = 0; w0 < n_words; w0 += kBitmapThreads) {
    const int w = w0 + tid;
    uint32_t bits = 0;
    if (w < n_words) {
      bits = bitmap[w];
      const int valid = K - 32 * w;  // columns of this word below K
      if (valid < 32) bits &= (1u << valid) - 1u;
    }
    const int c = __popc(bits);
    int incl = c;  // inclusive scan over the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    int before = 0, tile = 0;
    for (int k = 0; k < kBitmapThreads / 32; ++k) {
      const int t = warp_tot[k];
      before += k < warp ? t : 0;
      tile += t;
    }
    int pos = base + before + incl - c;
    while (bits) {
      const int b = __ffs(bits) - 1;
      bits &= bits - 1u;
      if (pos < max_s) idx[pos] = 32 * w + b;
      ++pos;
    }
    base += tile;
    __syncthreads();  // every thread has read warp_tot before the next tile rewrites it
  }
  if (tid == 0) *count = base;
}

// The index list as the bitmap (zeroed before): each index sets its bit; an index outside [0, K)
// or not above its predecessor sets *bad instead.
__global__ void qtea_index_to_bitmap_kernel(const int32_t* __restrict__ idx, int s, int K, uint32_t* bitmap,
                                            int* bad) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < s; i += gridDim.x * blockDim.x) {
    const int j = idx[i];
    if (j < 0 || j >= K || (i > 0 && idx[i - 1] >= j)) {
      atomicExch(bad, 1);
      continue;
    }
    atomicOr(bitmap + (j >> 5), 1u << (j & 31));
  }
}

cudaError_t launch_bitmap_to_index(const uint32_t* bitmap, int K, int32_t* idx, int max_s, int* count,
                                   cudaStream_t st) {
  qtea_bitmap_to_index_kernel<<<1, kBitmapThreads, 0, st>>>(bitmap, K, idx, max_s, count);
  return cudaGetLastError();
}

cudaError_t launch_index_to_bitmap(const int32_t* idx, int s, int K, uint32_t* bitmap, int* bad, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(bitmap, 0, sizeof(uint32_t) * (size_t)((K + 31) / 32), st);
  if (e != cudaSuccess || s == 0) return e;
  const int threads = 256;
  int blocks = (s + threads - 1) / threads;
  if (blocks > 1024) blocks = 1024;
  qtea_index_to_bitmap_kernel<<<blocks, threads, 0, st>>>(idx, s, K, bitmap, bad);
  return cudaGetLastError();
}

}  // namespace qtea
