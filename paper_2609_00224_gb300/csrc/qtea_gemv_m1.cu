// Batch-1 QTEA GEMV for sm_103a: y = alpha * (T . (v*x)) + sparse 1:4 residual, for one or
// several independent problems in one launch.
//
// Computes Eq. 10 (one alpha per row, beta = 0) plus Eq. 11 of the QTEA paper (Sec. 3.5).
// Design:
//  * Grouped persistent stream-K: the (problem, 512-row tile, 512-column chunk) units of all
//    problems form one sequence; one CTA per SM takes an equal contiguous share, so every SM
//    streams the same number of weight bytes and one launch amortises its fixed costs over
//    all problems.
//  * TMA ring: a producer lane fetches each unit as two 256 x 128-byte boxes of packed 2-bit
//    codes (cp.async.bulk.tensor, 128-byte swizzle) into a shared-memory ring guarded by
//    mbarriers; eight consumer warps decode from shared memory, each lane owning two rows,
//    so no cross-lane reduction is needed.
//  * Decode: v*x (the column rescale of Sec. 3.3, fused into activation staging as the
//    paper fuses it into its LUT precompute) is held per 512-column chunk as 24-bit fixed
//    point split into three byte planes. Codes are masked four at a time into byte lanes and
//    multiplied with dp4a, so sum_j c_j X_j is exact in integers; the ternary value is
//    c - 1, whose contribution is removed with the chunk's sum of X.
//  * Residual (Eq. 11): each CTA adds sum_c R x_{S_c} for the salient columns inside the
//    chunks it decodes (located by binary search of the sorted salient list), so the
//    residual work is spread like the weight stream; its loads are issued before the unit's
//    decode to hide their latency. The values are never scaled by alpha or v.
//  * Split tiles are reduced by the last-arriving CTA (atomic counter, no spin-wait) in a
//    fixed CTA order, so results are bitwise reproducible.
// Every wait on an mbarrier is bounded: after ~2 s the waiting thread records
// QTEA_ERR_TIMEOUT in the status word and the CTA abandons its work.
#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr unsigned long long kWaitLimitNs = 2000000000ull;
constexpr int kResPrefetch = 8;  // residual entries per lane loaded ahead of a unit's decode

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{ .reg .b64 st; mbarrier.arrive.shared::cta.b64 st, [%0]; }" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("{ .reg .b64 st; mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1; }" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait until the phase with the given parity has completed; false after the time limit.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0 && global_ns() - t0 > kWaitLimitNs) {
      atomicExch(status, (int)QTEA_ERR_TIMEOUT);
      return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__device__ __forceinline__ float h2f(uint16_t b) { return __half2float(__ushort_as_half(b)); }

// CTA whose range contains unit u.
__device__ __forceinline__ int unit_owner(long long u, long long total, int grid) {
  return (int)(((u + 1) * grid - 1) / total);
}

// Accumulators of one row for one chunk: [plane][scale set]; scale set 0 holds codes of
// column groups 0 and 2 (weight 1), set 1 codes of groups 1 and 3 (weight 4).
template <int P>
struct RowAcc {
  int a[P][2];
};

// One 32-bit word = 16 codes of one row. Plane registers of the word, in the order
// [group k][plane q] (k = columns {k, 4+k, 8+k, 12+k} in byte lanes 0..3): for P = 3,
// P0 = {g0p0, g0p1, g0p2, g1p0}, P1 = {g1p1, g1p2, g2p0, g2p1}, P2 = {g2p2, g3p0, g3p1, g3p2};
// for P = 2, P0 = {g0p0, g0p1, g1p0, g1p1}, P1 = {g2p0, g2p1, g3p0, g3p1}. The top plane is
// signed, the others unsigned.
__device__ __forceinline__ void decode_word3(uint32_t w, const uint4& P0, const uint4& P1, const uint4& P2,
                                             RowAcc<3>& r) {
  const uint32_t w4 = w >> 4;
  const uint32_t g0 = w & 0x03030303u;   // columns 0,4,8,12 -> byte lanes, values 0..2
  const uint32_t g1 = w & 0x0C0C0C0Cu;   // columns 1,5,9,13, values 0,4,8
  const uint32_t g2 = w4 & 0x03030303u;  // columns 2,6,10,14
  const uint32_t g3 = w4 & 0x0C0C0C0Cu;  // columns 3,7,11,15
  r.a[0][0] = (int)__dp4a(g0, P0.x, (unsigned)r.a[0][0]);
  r.a[1][0] = (int)__dp4a(g0, P0.y, (unsigned)r.a[1][0]);
  r.a[2][0] = __dp4a((int)g0, (int)P0.z, r.a[2][0]);
  r.a[0][1] = (int)__dp4a(g1, P0.w, (unsigned)r.a[0][1]);
  r.a[1][1] = (int)__dp4a(g1, P1.x, (unsigned)r.a[1][1]);
  r.a[2][1] = __dp4a((int)g1, (int)P1.y, r.a[2][1]);
  r.a[0][0] = (int)__dp4a(g2, P1.z, (unsigned)r.a[0][0]);
  r.a[1][0] = (int)__dp4a(g2, P1.w, (unsigned)r.a[1][0]);
  r.a[2][0] = __dp4a((int)g2, (int)P2.x, r.a[2][0]);
  r.a[0][1] = (int)__dp4a(g3, P2.y, (unsigned)r.a[0][1]);
  r.a[1][1] = (int)__dp4a(g3, P2.z, (unsigned)r.a[1][1]);
  r.a[2][1] = __dp4a((int)g3, (int)P2.w, r.a[2][1]);
}

__device__ __forceinline__ void decode_word2(uint32_t w, const uint4& P0, const uint4& P1, RowAcc<2>& r) {
  const uint32_t w4 = w >> 4;
  const uint32_t g0 = w & 0x03030303u;
  const uint32_t g1 = w & 0x0C0C0C0Cu;
  const uint32_t g2 = w4 & 0x03030303u;
  const uint32_t g3 = w4 & 0x0C0C0C0Cu;
  r.a[0][0] = (int)__dp4a(g0, P0.x, (unsigned)r.a[0][0]);
  r.a[1][0] = __dp4a((int)g0, (int)P0.y, r.a[1][0]);
  r.a[0][1] = (int)__dp4a(g1, P0.z, (unsigned)r.a[0][1]);
  r.a[1][1] = __dp4a((int)g1, (int)P0.w, r.a[1][1]);
  r.a[0][0] = (int)__dp4a(g2, P1.x, (unsigned)r.a[0][0]);
  r.a[1][0] = __dp4a((int)g2, (int)P1.y, r.a[1][0]);
  r.a[0][1] = (int)__dp4a(g3, P1.z, (unsigned)r.a[0][1]);
  r.a[1][1] = __dp4a((int)g3, (int)P1.w, r.a[1][1]);
}

// 4 * sum_j (c_j - 1) X_j over the chunk, exact, as int64.
template <int P>
__device__ __forceinline__ long long finish_chunk(const RowAcc<P>& r, long long sum_x) {
  long long v = 0;
#pragma unroll
  for (int q = 0; q < P; ++q) v += (4ll * r.a[q][0] + r.a[q][1]) * (1ll << (8 * q));
  return v - 4ll * sum_x;
}

// Decode one unit (two rows per lane, 32 words each) against the chunk's P byte planes.
// The next word's planes and the next 16 bytes of both rows are loaded while the current
// word decodes.
template <int P>
__device__ __forceinline__ void decode_unit(const uint4* row0, const uint4* row1, const uint4* pl, int sw,
                                            RowAcc<P>& a0, RowAcc<P>& a1) {
  constexpr int kW = (P == 3) ? 3 : 2;  // uint4 of planes per word (stride 3 in the slot)
#pragma unroll
  for (int k = 0; k < P; ++k) { a0.a[k][0] = a0.a[k][1] = 0; a1.a[k][0] = a1.a[k][1] = 0; }
  uint4 P0 = pl[0], P1 = pl[1], P2 = kW == 3 ? pl[2] : make_uint4(0, 0, 0, 0);
  uint4 c0 = row0[0 ^ sw], c1 = row1[0 ^ sw];
#pragma unroll 1
  for (int jj = 0; jj < 8; ++jj) {
    const uint4 n0 = row0[((jj + 1) & 7) ^ sw];
    const uint4 n1 = row1[((jj + 1) & 7) ^ sw];
    const uint32_t w0[4] = {c0.x, c0.y, c0.z, c0.w};
    const uint32_t w1[4] = {c1.x, c1.y, c1.z, c1.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int nw = ((4 * jj + e + 1) & 31) * 3;
      const uint4 Q0 = pl[nw], Q1 = pl[nw + 1];
      const uint4 Q2 = kW == 3 ? pl[nw + 2] : make_uint4(0, 0, 0, 0);
      if constexpr (P == 3) {
        decode_word3(w0[e], P0, P1, P2, a0);
        decode_word3(w1[e], P0, P1, P2, a1);
      } else {
        decode_word2(w0[e], P0, P1, a0);
        decode_word2(w1[e], P0, P1, a1);
      }
      P0 = Q0;
      P1 = Q1;
      P2 = Q2;
    }
    c0 = n0;
    c1 = n1;
  }
}

__device__ __forceinline__ void add_residual(float (&rp)[4], uint16_t rv, uint8_t rb, int c, float xv) {
  const int pos = (rb >> (2 * (c & 3))) & 3;
  const float val = h2f(rv) * xv;
  rp[0] += pos == 0 ? val : 0.f;
  rp[1] += pos == 1 ? val : 0.f;
  rp[2] += pos == 2 ? val : 0.f;
  rp[3] += pos == 3 ? val : 0.f;
}

// Activation staging of one 512-column chunk by one warp, 16 columns per lane, in two steps
// so that the loads of every chunk can be issued before the weight stream starts.
struct ChunkLoads {
  uint32_t x[8], v[8];  // fp16 pairs of columns 16*lane .. 16*lane+15 (zero beyond K)
};

__device__ __noinline__ void load_chunk(const ProblemArgs& a, int ch, int lane, ChunkLoads& L) {
  const int col0 = ch * kChunkCols + lane * 16;
  const bool vec_ok = ((reinterpret_cast<uintptr_t>(a.x) | reinterpret_cast<uintptr_t>(a.v)) & 15) == 0;
  if (vec_ok && col0 + 16 <= a.K) {
    const uint4* xv4 = reinterpret_cast<const uint4*>(a.x + col0);
    const uint4* vv4 = reinterpret_cast<const uint4*>(a.v + col0);
    const uint4 xa = __ldg(xv4), xb = __ldg(xv4 + 1), va = __ldg(vv4), vb = __ldg(vv4 + 1);
    L.x[0] = xa.x; L.x[1] = xa.y; L.x[2] = xa.z; L.x[3] = xa.w;
    L.x[4] = xb.x; L.x[5] = xb.y; L.x[6] = xb.z; L.x[7] = xb.w;
    L.v[0] = va.x; L.v[1] = va.y; L.v[2] = va.z; L.v[3] = va.w;
    L.v[4] = vb.x; L.v[5] = vb.y; L.v[6] = vb.z; L.v[7] = vb.w;
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int c = col0 + 2 * i;
      const uint32_t x0 = c < a.K ? a.x[c] : 0u, x1 = c + 1 < a.K ? a.x[c + 1] : 0u;
      const uint32_t v0 = c < a.K ? a.v[c] : 0u, v1 = c + 1 < a.K ? a.v[c + 1] : 0u;
      L.x[i] = x0 | (x1 << 16);
      L.v[i] = v0 | (v1 << 16);
    }
  }
}

// Planes, scale, sum of X, salient range and x at the chunk's first kChunkSalCap salient
// columns (gathered from the lanes' registers), written to one shared-memory slot.
__device__ __noinline__ void compute_chunk(const ProblemArgs& a, int ch, const ChunkLoads& L, uint8_t* slot,
                                              const int* salc, int lane) {
  float xt[16];
#pragma unroll
  for (int i = 0; i < 8; ++i) {  // exact: fp16 x fp16 fits fp32
    xt[2 * i] = h2f((uint16_t)(L.v[i] & 0xffffu)) * h2f((uint16_t)(L.x[i] & 0xffffu));
    xt[2 * i + 1] = h2f((uint16_t)(L.v[i] >> 16)) * h2f((uint16_t)(L.x[i] >> 16));
  }
  float amax = 0.f, ssq = 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    amax = fmaxf(amax, fabsf(xt[i]));
    ssq = fmaf(xt[i], xt[i], ssq);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    ssq += __shfl_xor_sync(0xffffffffu, ssq, o);
  }
  // 16-bit fixed point only where the chunk's largest |v*x| is within 8x its root mean square
  // (no outliers that would coarsen the quantum of the others); otherwise 24-bit
  const bool two = a.act_bits == 16 && amax * amax <= 64.f * (ssq / (float)kChunkCols);
  // amax in [2^e, 2^(e+1)) -> q = 2^(e-21), |X| <= 2^22 (24-bit) or q = 2^(e-13), |X| <= 2^14
  const int e = amax > 0.f ? (int)((__float_as_uint(amax) >> 23) & 0xff) - 127 : 0;
  const int qsh = two ? 13 : 21;
  const float inv_q = __uint_as_float((uint32_t)(127 + qsh - e) << 23);
  int X[16];
  long long sx = 0;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    X[i] = __float2int_rn(xt[i] * inv_q);
    sx += X[i];
  }
  uint4* dst = reinterpret_cast<uint4*>(slot + (size_t)lane * kPlaneBytesPerWord);
  if (two) {
    uint32_t reg[8];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        uint32_t r = 0;
#pragma unroll
        for (int bb = 0; bb < 4; ++bb) r |= ((uint32_t)(X[4 * bb + k] >> (8 * q)) & 0xffu) << (8 * bb);
        reg[k * 2 + q] = r;
      }
    }
    dst[0] = make_uint4(reg[0], reg[1], reg[2], reg[3]);
    dst[1] = make_uint4(reg[4], reg[5], reg[6], reg[7]);
  } else {
    uint32_t reg[12];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        uint32_t r = 0;
#pragma unroll
        for (int bb = 0; bb < 4; ++bb) r |= ((uint32_t)(X[4 * bb + k] >> (8 * q)) & 0xffu) << (8 * bb);
        reg[k * 3 + q] = r;
      }
    }
    dst[0] = make_uint4(reg[0], reg[1], reg[2], reg[3]);
    dst[1] = make_uint4(reg[4], reg[5], reg[6], reg[7]);
    dst[2] = make_uint4(reg[8], reg[9], reg[10], reg[11]);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) sx += __shfl_xor_sync(0xffffffffu, sx, o);
  // salient entries with column in [512 ch, 512 ch + 512): lanes 0 and 1 search the two bounds
  int bound = 0;
  if (lane < 2) {
    const int lim = (ch + lane) * kChunkCols;
    int lo = 0, hi = a.s;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (salc[mid] < lim) lo = mid + 1;
      else hi = mid;
    }
    bound = lo;
  }
  const int c_lo = __shfl_sync(0xffffffffu, bound, 0);
  const int c_hi = max(__shfl_sync(0xffffffffu, bound, 1), c_lo);
  const int n_xs = min(c_hi - c_lo, kChunkSalCap);
  // x at salient column j lives in lane (j mod 512) / 16, element j mod 16
  float* xs = reinterpret_cast<float*>(slot + kPlaneBytesPerChunk + sizeof(ChunkMeta));
#pragma unroll
  for (int r = 0; r < kChunkSalCap / 32; ++r) {
    const int idx = lane + 32 * r;
    int col = idx < n_xs ? salc[c_lo + idx] - ch * kChunkCols : 0;
    col = col < 0 ? 0 : (col > kChunkCols - 1 ? kChunkCols - 1 : col);
    const int src = col >> 4, word = (col & 15) >> 1;
    uint32_t got = 0;
#pragma unroll
    for (int w = 0; w < 8; ++w) {
      const uint32_t v = __shfl_sync(0xffffffffu, L.x[w], src);
      got = (w == word) ? v : got;
    }
    if (idx < n_xs) xs[idx] = h2f((uint16_t)((col & 1) ? (got >> 16) : (got & 0xffffu)));
  }
  if (lane == 0) {
    ChunkMeta mm;
    mm.scale4 = __uint_as_float((uint32_t)(127 + e - qsh - 2) << 23);  // q / 4
    mm.c_lo = c_lo;
    mm.c_hi = c_hi;
    mm.planes = two ? 2 : 3;
    mm.sum_x = sx;
    mm.pad2 = 0;
    *reinterpret_cast<ChunkMeta*>(slot + kPlaneBytesPerChunk) = mm;
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    qtea_gemv_m1_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ GroupParams gp) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int grid = gridDim.x;
  const int b = blockIdx.x;
  const int S = gp.n_stages;
  const int NP = gp.n_problems;

  // ---- prologue 1: the problem table is copied to shared memory by all threads at once (its
  //      first reads would otherwise be a chain of constant-cache misses); the copy sits in the
  //      ring, which no copy has been issued into yet
  ProblemArgs* prob = reinterpret_cast<ProblemArgs*>(smem);
  {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(gp.prob);
    uint32_t* dst = reinterpret_cast<uint32_t*>(prob);
    const int words = NP * (int)(sizeof(ProblemArgs) / 4);
    for (int i = threadIdx.x; i < words; i += blockDim.x) dst[i] = src[i];
  }
  if (warp == kProducerWarp && lane < NP)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.m[lane])) : "memory");
  const int u0 = gp.cta_u0[b], u1 = gp.cta_u0[b + 1];
  const int n_units = u1 - u0;
  __syncthreads();

  // ---- prologue 2: thread 0 plans shared memory (chunk slots, salient indices, residual ring,
  //      barriers); every thread derives the plan's offsets from the shared copy
  size_t misc_off = 0;
  int n_slots = 0;
  cta_smem_plan(prob, NP, S, u0, u1, nullptr, &n_slots, &misc_off);
  float* rsum = reinterpret_cast<float*>(smem + misc_off);  // per-warp gather of residual sums
  StageSlot* slots = reinterpret_cast<StageSlot*>(smem + misc_off + kResidFloats * sizeof(float));
  uint64_t* bars = reinterpret_cast<uint64_t*>(slots + kMaxProblems);
  uint64_t* full = bars;
  uint64_t* empty = bars + S;
  if (threadIdx.x == 0) {
    cta_smem_plan(prob, NP, S, u0, u1, slots, nullptr, nullptr);
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_u32(&full[i]), 1);                // producer arrival + TMA bytes
      mbar_init(smem_u32(&empty[i]), kConsumerWarps);  // one arrival per consumer warp
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();
  // per-problem values the loops need, out of the shared copy into registers
  int p_ub[kMaxProblems], p_nc[kMaxProblems];
#pragma unroll
  for (int p = 0; p < kMaxProblems; ++p) {
    p_ub[p] = p < NP ? (int)prob[p].unit_begin : 0x7fffffff;
    p_nc[p] = p < NP ? prob[p].n_chunks : 1;
  }

  // ---- prologue 3: issue the loads of the salient indices and of the activations of every
  //      chunk this CTA touches (one warp per chunk, kBatch chunks per warp in flight) before the
  //      weight stream competes with them for memory bandwidth
  constexpr int kBatch = 4;
  constexpr int kSalPerThread = 8;
  constexpr int kStageWarps = kConsumerWarps + 1;
  int n_items = 0;
  for (int j = 0; j < n_slots; ++j) n_items += slots[j].n_ch;
  // the salient index loads go to registers with compile-time indices (a dynamically indexed
  // array would live in local memory and every store would wait for its load)
  int s_tot = 0;
  for (int j = 0; j < n_slots; ++j) s_tot += slots[j].s;
  auto sal_load = [&](int e) -> int {
    int j = 0;
    while (j + 1 < n_slots && e >= slots[j].s) {
      e -= slots[j].s;
      ++j;
    }
    return gp.prob[slots[j].p].sal[e];
  };
  int sal_val[kSalPerThread];
#pragma unroll
  for (int k2 = 0; k2 < kSalPerThread; ++k2) {
    const int e = threadIdx.x + k2 * blockDim.x;
    sal_val[k2] = e < s_tot ? sal_load(e) : 0;
  }
  auto item_of = [&](int item, int& j, int& k) {
    j = 0;
    while (j + 1 < n_slots && item >= slots[j].n_ch) {
      item -= slots[j].n_ch;
      ++j;
    }
    k = item;
  };
  ChunkLoads L[kBatch];
#pragma unroll 1
  for (int r = 0; r < kBatch; ++r) {
    const int item = warp + r * kStageWarps;
    if (item < n_items) {
      int j, k;
      item_of(item, j, k);
      const ProblemArgs& a = prob[slots[j].p];
      int ch = slots[j].ch_start + k;
      if (ch >= a.n_chunks) ch -= a.n_chunks;
      load_chunk(a, ch, lane, L[r]);
    }
  }

  // unit cursor: problem, tile, chunk, slot and slot-local chunk, advanced without division
  struct Cursor {
    int p, t, ch, j, li;
  };
  Cursor start;
  {
    int p = 0;
    while (p + 1 < NP && u0 >= p_ub[p + 1]) ++p;
    const int v0 = u0 - p_ub[p];
    start.p = p;
    start.t = v0 / p_nc[p];
    start.ch = v0 - start.t * p_nc[p];
    start.j = 0;
    start.li = 0;
  }
  auto advance = [&](Cursor& c, int u_next) {
    const int nc = p_nc[c.p];
    if (++c.ch == nc) {
      c.ch = 0;
      ++c.t;
    }
    if (++c.li == nc) c.li = 0;
    if (c.p + 1 < NP && u_next >= p_ub[c.p + 1]) {
      ++c.p;
      c.t = 0;
      c.ch = 0;
      c.li = 0;
      while (c.j + 1 < n_slots && slots[c.j].p != c.p) ++c.j;
    }
  };
  // every field the loops read from the problem table is kept in registers or re-read from
  // the kernel parameters below, so the ring may be overwritten once everyone is past here
  __syncthreads();

  // ---- the first ring fills go out now, behind the staging loads
  auto issue = [&](const Cursor& c, int st) {
    const uint32_t bar = smem_u32(&full[st]);
    const uint32_t dst = smem_u32(smem + (size_t)st * kStageBytes);
    mbar_arrive_expect_tx(bar, kStageBytes);
    tma_load_2d(dst, &maps.m[c.p], c.ch * kChunkRowBytes, c.t * kTileRows, bar);
    tma_load_2d(dst + kBoxBytes, &maps.m[c.p], c.ch * kChunkRowBytes, c.t * kTileRows + kBoxRows, bar);
  };
  if (warp == kProducerWarp && lane == 0) {
    Cursor c = start;
    for (int i = 0; i < n_units && i < S; ++i) {
      issue(c, i);
      advance(c, u0 + i + 1);
    }
  }

  // ---- prologue 4: salient indices to shared memory, then the planes of every chunk
  {
    auto sal_store = [&](int e, int col) {
      int j = 0;
      while (j + 1 < n_slots && e >= slots[j].s) {
        e -= slots[j].s;
        ++j;
      }
      const int K = gp.prob[slots[j].p].K;
      reinterpret_cast<int*>(smem + slots[j].salc)[e] = col < 0 ? 0 : (col >= K ? K - 1 : col);
    };
#pragma unroll
    for (int k2 = 0; k2 < kSalPerThread; ++k2) {
      const int e = threadIdx.x + k2 * blockDim.x;
      if (e < s_tot) sal_store(e, sal_val[k2]);
    }
    for (int e = threadIdx.x + kSalPerThread * blockDim.x; e < s_tot; e += blockDim.x) sal_store(e, sal_load(e));
  }
  __syncthreads();
  for (int r0 = 0; r0 * kStageWarps < n_items; r0 += kBatch) {
#pragma unroll 1
    for (int r = 0; r < kBatch; ++r) {
      const int item = warp + (r0 + r) * kStageWarps;
      if (item < n_items) {
        int j, k;
        item_of(item, j, k);
        const ProblemArgs& a = gp.prob[slots[j].p];
        int ch = slots[j].ch_start + k;
        if (ch >= a.n_chunks) ch -= a.n_chunks;
        if (r0 > 0) load_chunk(a, ch, lane, L[r]);  // chunks beyond the first batch (long ranges)
        compute_chunk(a, ch, L[r], smem + slots[j].chunks + (size_t)k * kSlotBytes,
                      reinterpret_cast<const int*>(smem + slots[j].salc), lane);
      }
    }
  }
  __syncthreads();

  // ---------------------------------------------------------------- producer: the TMA ring
  if (warp == kProducerWarp) {
    if (lane != 0) return;
    Cursor c = start;
    int st = 0, ph = 0;  // stage and its fill parity
    int i = 0;
    bool ok = true;
    for (; i < n_units; ++i) {
      if (i >= S) {
        // wait until the consumers released the previous fill of this stage
        if (!mbar_wait(smem_u32(&empty[st]), (uint32_t)(ph ^ 1), gp.status)) {
          ok = false;
          break;
        }
        issue(c, st);
      }
      advance(c, u0 + i + 1);
      if (++st == S) {
        st = 0;
        ph ^= 1;
      }
    }
    // drain: no bulk copy may still be writing shared memory when the CTA exits
    const int n_issued = ok ? n_units : i;
    for (int s2 = 0; s2 < S && s2 < n_issued; ++s2) {
      const int fills = (n_issued - s2 + S - 1) / S;  // fills of stage s2
      if (!mbar_wait(smem_u32(&full[s2]), (uint32_t)((fills - 1) & 1), gp.status)) break;
    }
    return;
  }

  // ---------------------------------------------------------------- consumers: decode
  const int ra = warp * 64 + lane;  // tile rows owned by this lane: ra and ra + 32
  const int sw = lane & 7;          // 128-byte swizzle phase of both rows
  const int g = lane & 15, half = lane >> 4;  // residual work: group g of the warp's 16, parity half
  float yacc0 = 0.f, yacc1 = 0.f;
  float rp[4] = {0.f, 0.f, 0.f, 0.f};
  Cursor c = start;
  int st = 0, ph = 0;
  const long long total = gp.total_units;

  for (int i = 0; i < n_units; ++i) {
    const int u = u0 + i;
    const StageSlot& sl = slots[c.j];
    const uint8_t* slot = smem + sl.chunks + (size_t)c.li * kSlotBytes;

    // this unit's residual entries (salient columns inside the chunk, rows of the lane's
    // group) are loaded before the decode and used after it
    const ProblemArgs& a = gp.prob[c.p];
    const ChunkMeta m = *reinterpret_cast<const ChunkMeta*>(slot + kPlaneBytesPerChunk);
    const int rs = (a.s + 3) >> 2;
    const int q = (c.t * kTileRows + warp * 64) / 4 + g;
    const bool q_ok = q < (a.N >> 2);
    const uint16_t* rvq = a.rvals + (size_t)q * a.s;
    const uint8_t* riq = a.ridx + (size_t)q * rs;
    uint16_t pre_v[kResPrefetch];
    uint8_t pre_b[kResPrefetch];
#pragma unroll
    for (int k = 0; k < kResPrefetch; ++k) {
      const int cc = m.c_lo + half + 2 * k;
      const bool okk = q_ok && cc < m.c_hi;
      pre_v[k] = okk ? __ldg(rvq + cc) : (uint16_t)0;
      pre_b[k] = okk ? __ldg(riq + (cc >> 2)) : (uint8_t)0;
    }

    bool failed = !mbar_wait(smem_u32(&full[st]), (uint32_t)ph, gp.status);
    // all lanes agree on failure before touching the data or the barriers
    if (__any_sync(0xffffffffu, failed)) break;

    const uint4* row0 = reinterpret_cast<const uint4*>(smem + (size_t)st * kStageBytes + (size_t)ra * kChunkRowBytes);
    const uint4* row1 = row0 + 32 * (kChunkRowBytes / 16);
    const uint4* pl = reinterpret_cast<const uint4*>(slot);
    long long d0, d1;
    if (m.planes == 2) {
      RowAcc<2> a0, a1;
      decode_unit<2>(row0, row1, pl, sw, a0, a1);
      d0 = finish_chunk<2>(a0, m.sum_x);
      d1 = finish_chunk<2>(a1, m.sum_x);
    } else {
      RowAcc<3> a0, a1;
      decode_unit<3>(row0, row1, pl, sw, a0, a1);
      d0 = finish_chunk<3>(a0, m.sum_x);
      d1 = finish_chunk<3>(a1, m.sum_x);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&empty[st]));  // release the stage to the producer

    yacc0 += (float)d0 * m.scale4;
    yacc1 += (float)d1 * m.scale4;

    // residual (Eq. 11) of the unit's salient columns, unscaled by alpha and v
    {
      const float* xs = reinterpret_cast<const float*>(slot + kPlaneBytesPerChunk + sizeof(ChunkMeta));
      const int* salc = reinterpret_cast<const int*>(smem + sl.salc);
#pragma unroll
      for (int k = 0; k < kResPrefetch; ++k) {
        const int cc = m.c_lo + half + 2 * k;
        if (q_ok && cc < m.c_hi) {
          const float xv = (cc - m.c_lo < kChunkSalCap) ? xs[cc - m.c_lo] : h2f(__ldg(a.x + salc[cc]));
          add_residual(rp, pre_v[k], pre_b[k], cc, xv);
        }
      }
      if (q_ok) {
        for (int cc = m.c_lo + 2 * kResPrefetch + half; cc < m.c_hi; cc += 2) {
          const float xv = (cc - m.c_lo < kChunkSalCap) ? xs[cc - m.c_lo] : h2f(__ldg(a.x + salc[cc]));
          add_residual(rp, __ldg(rvq + cc), __ldg(riq + (cc >> 2)), cc, xv);
        }
      }
    }

    // ---- tile epilogue once this CTA's part of tile t is done
    if (c.ch == p_nc[c.p] - 1 || u == u1 - 1) {
      const int t = c.t;
      const long long A = (long long)p_ub[c.p] + (long long)t * p_nc[c.p], B = A + p_nc[c.p];
      // per-row residual sums: lane (g, half) holds positions 0..3 of group g; gather by row
      float* rw = rsum + (size_t)warp * (16 * 2 * 4);
#pragma unroll
      for (int k = 0; k < 4; ++k) rw[(g * 2 + half) * 4 + k] = rp[k];
      __syncwarp();
      // row ra of the warp is local row `lane` -> group lane/4, position lane%4; ra+32 -> group 8 + lane/4
      const float res0 = rw[((lane >> 2) * 2 + 0) * 4 + (lane & 3)] + rw[((lane >> 2) * 2 + 1) * 4 + (lane & 3)];
      const float res1 =
          rw[((8 + (lane >> 2)) * 2 + 0) * 4 + (lane & 3)] + rw[((8 + (lane >> 2)) * 2 + 1) * 4 + (lane & 3)];
      __syncwarp();
      rp[0] = rp[1] = rp[2] = rp[3] = 0.f;
      const int row0g = t * kTileRows + ra, row1g = row0g + 32;
      const float al0 = row0g < a.N ? h2f(a.alpha[row0g]) : 0.f;
      const float al1 = row1g < a.N ? h2f(a.alpha[row1g]) : 0.f;
      const float val0 = al0 * yacc0 + res0;
      const float val1 = al1 * yacc1 + res1;
      if (A >= u0 && B <= u1) {
        if (row0g < a.N) a.y[row0g] = val0;
        if (row1g < a.N) a.y[row1g] = val1;
      } else {
        // partial tile: publish this warp's 64 rows, then the last of the tile's contributors
        // (per warp: counter t * kConsumerWarps + warp) sums all partials in CTA order. Slot 0
        // of a CTA holds the tile its range starts in, slot 1 the tile its range ends in.
        const int my_slot = (u0 >= A) ? 0 : 1;
        float* wsp = a.ws + ((size_t)b * 2 + my_slot) * kTileRows;
        wsp[ra] = val0;
        wsp[ra + 32] = val1;
        __threadfence();
        __syncwarp();
        const int bf = unit_owner(A, total, grid), bl = unit_owner(B - 1, total, grid);
        int last = 0;
        if (lane == 0) {
          unsigned* ctr = a.counters + (size_t)t * kConsumerWarps + warp;
          const unsigned prev = atomicAdd(ctr, 1u);
          last = (prev == (unsigned)(bl - bf));  // every CTA in [bf, bl] holds units of this tile
          if (last) {
            __threadfence();
            *ctr = 0u;  // self-reset for the next call
          }
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          float s0 = 0.f, s1 = 0.f;
          for (int cb = bf; cb <= bl; ++cb) {
            const int cslot = (gp.cta_u0[cb] >= A) ? 0 : 1;
            const float* src = a.ws + ((size_t)cb * 2 + cslot) * kTileRows;
            s0 += __ldcg(src + ra);
            s1 += __ldcg(src + ra + 32);
          }
          if (row0g < a.N) a.y[row0g] = s0;
          if (row1g < a.N) a.y[row1g] = s1;
        }
      }
      yacc0 = 0.f;
      yacc1 = 0.f;
    }
    advance(c, u + 1);
    if (++st == S) {
      st = 0;
      ph ^= 1;
    }
  }
}

}  // namespace

// Allow the kernel the largest dynamic shared memory the device grants next to its static
// shared memory; *dyn_max receives that size.
cudaError_t m1_configure(size_t smem_optin, size_t* dyn_max) {
  cudaFuncAttributes attr;
  cudaError_t e = cudaFuncGetAttributes(&attr, qtea_gemv_m1_kernel);
  if (e != cudaSuccess) return e;
  const size_t dyn = smem_optin > attr.sharedSizeBytes ? smem_optin - attr.sharedSizeBytes : 0;
  *dyn_max = dyn;
  return cudaFuncSetAttribute(qtea_gemv_m1_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
}

cudaError_t launch_m1(const TensorMaps& maps, const GroupParams& p, int grid, size_t smem, cudaStream_t st) {
  qtea_gemv_m1_kernel<<<grid, kThreads, smem, st>>>(maps, p);
  return cudaGetLastError();
}

}  // namespace qtea
