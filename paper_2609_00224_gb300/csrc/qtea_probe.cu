// Issue rates behind the decode choice of the batch-1 kernels (a diagnostic; no step of the path).
//
// The batch-1 decode could run on the dp4a pipe (the current kernels) or on the tensor cores through
// mma.sync, with A built from the 2-bit codes in registers. What decides between them is the rate at
// which each instruction issues when its operands change every time, as they do in a decode. Each
// kernel below runs 8 warps per SM, every warp 8 independent accumulator chains, and reports clock64
// cycles per instruction per sub-partition (4 per SM):
//   0  mma.sync m16n8k16 f16 -> f32, A and B constant
//   1  mma.sync m16n8k16 f16 -> f32, A masked from a word that changes every instruction (fp16
//      subnormal code values, the form a decode of 2-bit codes gives)
//   2  mma.sync m16n8k32 e4m3 -> f32, A and B constant
//   3  mma.sync m16n8k32 e4m3 -> f32, A masked from a word that changes every instruction
//   4  dp4a, four per chain step
// For batch 1 a m16n8k16 MMA does 256 useful multiply-adds (one of its 8 columns), a m16n8k32 MMA 512,
// a dp4a 4 byte products (2 weights at 16-bit activations).
#include <cuda_runtime.h>
#include <stdint.h>

#include "qtea.h"

namespace qtea {
namespace {

constexpr int kProbeWarps = 8;
constexpr int kProbeIters = 2000;

template <int KIND>
__global__ void __launch_bounds__(kProbeWarps * 32, 1) probe_kernel(uint32_t seed, float* sink, long long* cycles) {
  uint32_t a0 = seed * 3u + threadIdx.x, a1 = a0 ^ 0x11111111u, a2 = a0 ^ 0x22222222u, a3 = a0 ^ 0x33333333u;
  uint32_t b0 = seed ^ 0x01010101u, b1 = seed ^ 0x02020202u;
  if (KIND == 0 || KIND == 1) {  // small fp16 values
    a0 &= 0x00ff00ffu; a1 &= 0x00ff00ffu; a2 &= 0x00ff00ffu; a3 &= 0x00ff00ffu; b0 &= 0x00ff00ffu; b1 &= 0x00ff00ffu;
  } else if (KIND == 2 || KIND == 3) {  // small e4m3 values
    a0 &= 0x07070707u; a1 &= 0x07070707u; a2 &= 0x07070707u; a3 &= 0x07070707u; b0 &= 0x07070707u; b1 &= 0x07070707u;
  }
  float d[8][4];
  int di[8][4];
#pragma unroll
  for (int c = 0; c < 8; ++c)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      d[c][j] = 0.f;
      di[c][j] = 0;
    }
  __syncthreads();
  const long long t0 = clock64();
  for (int it = 0; it < kProbeIters; ++it) {
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      if (KIND == 0) {
        asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                     : "+f"(d[c][0]), "+f"(d[c][1]), "+f"(d[c][2]), "+f"(d[c][3])
                     : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
      } else if (KIND == 1) {
        const uint32_t w = a0 * (uint32_t)(it * 8 + c) + b1;
        asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                     : "+f"(d[c][0]), "+f"(d[c][1]), "+f"(d[c][2]), "+f"(d[c][3])
                     : "r"(w & 0x00030003u), "r"(w & 0x000C000Cu), "r"(w & 0x00300030u), "r"(w & 0x00C000C0u),
                       "r"(b0), "r"(b1));
      } else if (KIND == 2) {
        asm volatile("mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                     : "+f"(d[c][0]), "+f"(d[c][1]), "+f"(d[c][2]), "+f"(d[c][3])
                     : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
      } else if (KIND == 3) {
        const uint32_t w = a0 * (uint32_t)(it * 8 + c) + b1;
        const uint32_t t = __umulhi(w, 1u << 28);
        asm volatile("mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                     : "+f"(d[c][0]), "+f"(d[c][1]), "+f"(d[c][2]), "+f"(d[c][3])
                     : "r"(w & 0x03030303u), "r"(w & 0x0C0C0C0Cu), "r"(t & 0x03030303u), "r"(t & 0x0C0C0C0Cu),
                       "r"(b0), "r"(b1));
      } else {
        di[c][0] = __dp4a((int)a0, (int)b0, di[c][0]);
        di[c][1] = __dp4a((int)a1, (int)b0, di[c][1]);
        di[c][2] = __dp4a((int)a2, (int)b1, di[c][2]);
        di[c][3] = __dp4a((int)a3, (int)b1, di[c][3]);
      }
    }
  }
  __syncthreads();
  const long long t1 = clock64();
  float s = 0.f;
#pragma unroll
  for (int c = 0; c < 8; ++c)
#pragma unroll
    for (int j = 0; j < 4; ++j) s += d[c][j] + (float)di[c][j];
  sink[blockIdx.x * blockDim.x + threadIdx.x] = s;  // keeps the chains live
  if (threadIdx.x == 0) cycles[blockIdx.x] = t1 - t0;
}

template <int KIND>
cudaError_t run_probe(int grid, float* sink, long long* cycles, double* out) {
  probe_kernel<KIND><<<grid, kProbeWarps * 32>>>(12345u, sink, cycles);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  long long c = 0;
  if ((e = cudaMemcpy(&c, cycles, sizeof(c), cudaMemcpyDeviceToHost)) != cudaSuccess) return e;
  // instructions per sub-partition: iterations x 8 chains x (warps / 4), four dp4a per chain step
  const double per_smsp = (double)kProbeIters * 8 * kProbeWarps / 4 * (KIND == 4 ? 4 : 1);
  *out = (double)c / per_smsp;
  return cudaSuccess;
}

}  // namespace
}  // namespace qtea

extern "C" int qtea_probe_decode_rates(double* cycles_per_instruction, int n) {
  using namespace qtea;
  if (!cycles_per_instruction || n < 5) return QTEA_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  float* sink = nullptr;
  long long* cycles = nullptr;
  if (cudaMalloc(&sink, (size_t)sms * kProbeWarps * 32 * sizeof(float)) != cudaSuccess ||
      cudaMalloc(&cycles, (size_t)sms * sizeof(long long)) != cudaSuccess) {
    cudaGetLastError();
    if (sink) cudaFree(sink);
    return QTEA_ERR_ALLOC;
  }
  cudaError_t e = run_probe<0>(sms, sink, cycles, &cycles_per_instruction[0]);
  if (e == cudaSuccess) e = run_probe<1>(sms, sink, cycles, &cycles_per_instruction[1]);
  if (e == cudaSuccess) e = run_probe<2>(sms, sink, cycles, &cycles_per_instruction[2]);
  if (e == cudaSuccess) e = run_probe<3>(sms, sink, cycles, &cycles_per_instruction[3]);
  if (e == cudaSuccess) e = run_probe<4>(sms, sink, cycles, &cycles_per_instruction[4]);
  cudaFree(sink);
  cudaFree(cycles);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  return QTEA_OK;
}
