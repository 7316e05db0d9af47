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

}  // namespace qtea
