// General QTEA GEMV (any batch 1 <= M <= 16, any N, K): y = alpha * (T . (v*x)) + residual.
//
// Eq. 10 with one alpha per row and beta = 0, plus Eq. 11 (Sec. 3.5 of the QTEA paper).
// One warp per output row: lanes stride over the row's 16-column words of packed codes
// (coalesced 4-byte loads), decode each code to -1/0/+1 and accumulate T * (v*x) in fp32 for
// every batch row; v*x is formed exactly in fp32 from the fp16 inputs. The residual of the
// row's group of four is added by the same warp. This kernel serves M > 1 and shapes whose
// activation staging does not fit the batch-1 kernel's shared memory.
#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr int kGenWarps = 4;

template <int MB>
__global__ void __launch_bounds__(kGenWarps * 32) qtea_gemv_generic_kernel(const GenericParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int o = blockIdx.x * kGenWarps + warp;
  if (o >= p.N) return;
  const int M = p.M;
  float acc[MB], res[MB];
#pragma unroll
  for (int m = 0; m < MB; ++m) { acc[m] = 0.f; res[m] = 0.f; }

  const uint32_t* row = reinterpret_cast<const uint32_t*>(p.packed + (size_t)o * (p.K_pad / 4));
  const int n_words = (p.K + 15) / 16;
  for (int wi = lane; wi < n_words; wi += 32) {
    const uint32_t w = row[wi];
#pragma unroll 4
    for (int i = 0; i < 16; ++i) {
      const int col = wi * 16 + i;
      const int t = (int)((w >> (2 * i)) & 3u) - 1;
      if (t == 0 || col >= p.K) continue;
      const float vj = h2f(p.v[col]);
#pragma unroll
      for (int m = 0; m < MB; ++m) {
        if (m < M) {
          const float xv = vj * h2f(p.x[(size_t)m * p.K + col]);  // exact in fp32
          acc[m] += t > 0 ? xv : -xv;
        }
      }
    }
  }
  if (p.s > 0) {
    const int q = o >> 2, pos = o & 3, rs = (p.s + 3) / 4;
    for (int c = lane; c < p.s; c += 32) {
      if (((p.ridx[(size_t)q * rs + (c >> 2)] >> (2 * (c & 3))) & 3) != pos) continue;
      int j = p.sal[c];
      j = j < 0 ? 0 : (j >= p.K ? p.K - 1 : j);
      const float r = h2f(p.rvals[(size_t)q * p.s + c]);
#pragma unroll
      for (int m = 0; m < MB; ++m)
        if (m < M) res[m] += r * h2f(p.x[(size_t)m * p.K + j]);
    }
  }
  const float al = h2f(p.alpha[o]);
#pragma unroll
  for (int m = 0; m < MB; ++m) {
    float a = acc[m], r = res[m];
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      a += __shfl_xor_sync(0xffffffffu, a, off);
      r += __shfl_xor_sync(0xffffffffu, r, off);
    }
    if (lane == 0 && m < M) p.y[(size_t)m * p.N + o] = al * a + r;
  }
}

}  // namespace

cudaError_t launch_generic(const GenericParams& p, cudaStream_t st) {
  const int grid = (p.N + kGenWarps - 1) / kGenWarps;
  if (grid == 0) return cudaSuccess;
  const int threads = kGenWarps * 32;
  if (p.M <= 1) qtea_gemv_generic_kernel<1><<<grid, threads, 0, st>>>(p);
  else if (p.M <= 2) qtea_gemv_generic_kernel<2><<<grid, threads, 0, st>>>(p);
  else if (p.M <= 4) qtea_gemv_generic_kernel<4><<<grid, threads, 0, st>>>(p);
  else if (p.M <= 8) qtea_gemv_generic_kernel<8><<<grid, threads, 0, st>>>(p);
  else qtea_gemv_generic_kernel<16><<<grid, threads, 0, st>>>(p);
  return cudaGetLastError();
}

}  // namespace qtea
