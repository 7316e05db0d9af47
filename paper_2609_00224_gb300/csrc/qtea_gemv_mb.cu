// Low-batch QTEA GEMV for sm_103a (2 <= M <= 16): y[m] = alpha * (T . (v * x[m])) + residual,
// on the tensor cores.
//
// Computes Eq. 10 (one alpha per row, beta = 0) plus Eq. 11 of the QTEA paper (Sec. 3.5) for a
// batch of M activation rows. With M rows the product is a skinny dense contraction, so it runs
// on mma.sync m16n8k16 (fp16 operands, fp32 accumulation), exactly:
//  * A = T * v: the ternary code times the column rescale of Sec. 3.3. T is -1, 0 or +1 and v an
//    fp16 value, so every element of A is an fp16 value, formed in registers from the 2-bit codes
//    (byte permute, a multiply that spreads the byte, the 0x6400 magic exponent, two fp16 fix-ups
//    and a multiply by v).
//  * B = x, the fp16 activations, unchanged; each product A * B is exact in fp32 and the sums
//    accumulate in fp32.
//  * The residual of Eq. 11 is an exact contraction too: over "virtual columns", one per
//    salient column, A holds the fp16 residual value of the row's group where the stored
//    position is the row and 0 elsewhere, and B holds x at the salient column. It is accumulated
//    apart, since alpha does not scale it.
// Work: a unit is a 128-row tile. A cluster of C CTAs (C chosen so that tiles x C fills the GPU)
// shares a tile: CTA rank r takes chunks [r n/C, (r+1) n/C) and residual steps r, r + C, ...; the
// ranks' partial rows go through distributed shared memory into rank 0, which adds them in rank
// order (no partial sums in global memory, a fixed summation order). Eight consumer warps each
// own 16 rows of the tile; a producer lane streams the CTA's 512-column chunks through a ring of
// shared-memory stages by TMA: 128 rows x 128 bytes of codes (128-byte swizzle), the 16 x 512 block of x
// (128-byte swizzle, rows beyond M read as zero) and 512 values of v. x at the salient columns is
// gathered once per CTA. The k order inside each 16-column step is permuted so that a thread's
// four k slots are four consecutive columns, i.e. one byte of codes.
// Every wait on an mbarrier is bounded (~2 s, then QTEA_ERR_TIMEOUT in the status word).
#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr unsigned long long kWaitLimitNs = 2000000000ull;
constexpr int kMbConsumerWarps = 8;
constexpr int kMbThreads = (kMbConsumerWarps + 1) * 32;
constexpr int kMbTileRows = 128;
constexpr int kMbCodeBytes = kMbTileRows * kChunkRowBytes;  // 16384
constexpr int kMbXBoxCols = 64;                              // 128-byte rows of fp16
constexpr int kMbXBytes = 16 * kChunkCols * 2;               // 16384: 8 boxes of 16 x 64
constexpr int kMbVBytes = kChunkCols * 2;                    // 1024
constexpr int kMbStageBytes = 34816;                         // codes, x, v, rounded to 1024

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

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > kWaitLimitNs) {
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

__device__ __forceinline__ void mma_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t h2_as_u32(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u32_as_h2(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }

// The four codes of byte q of a code word as two fp16 pairs of T * v (columns 4q, 4q+1 and
// 4q+2, 4q+3 of the 16-column step): a code c = T + 1 is placed in the mantissa of 1024
// (0x6400), 1025 is subtracted (c in bits 0-1) or the value is scaled by 1/16 and 65 subtracted
// (c in bits 4-5), and the result, exactly -1, 0 or 1, multiplies v.
__device__ __forceinline__ void decode_byte(uint32_t word, uint32_t q, uint32_t v01, uint32_t v23, uint32_t& a01,
                                            uint32_t& a23) {
  const uint32_t b = __byte_perm(word, 0u, 0x4440u | q);  // byte q alone
  const uint32_t s = b * 0x4001u;                           // b in bits 0-7 and 14-21
  const uint32_t w01 = (s & 0x00030003u) | 0x64006400u;     // 1024 + c0 | 1024 + c1
  const uint32_t w23 = (s & 0x00300030u) | 0x64006400u;     // 1024 + 16 c2 | 1024 + 16 c3
  const __half2 t01 = __hsub2(u32_as_h2(w01), __float2half2_rn(1025.f));
  const __half2 t23 = __hfma2(u32_as_h2(w23), __float2half2_rn(0.0625f), __float2half2_rn(-65.f));
  a01 = h2_as_u32(__hmul2(t01, u32_as_h2(v01)));
  a23 = h2_as_u32(__hmul2(t23, u32_as_h2(v23)));
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t n_clusters() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void st_cluster_v4(uint32_t addr, float a, float b, float c, float d) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t remote_bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote_bar) : "memory");
}

// Wait for a phase completed by arrivals from other CTAs of the cluster (acquire at cluster scope).
__device__ __forceinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity, int* status) {
  const unsigned long long t0 = global_ns();
  for (;;) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    if (ok) return true;
    if (global_ns() - t0 > kWaitLimitNs) {
      atomicExch(status, (int)QTEA_ERR_TIMEOUT);
      return false;
    }
  }
}

// Shared memory of the kernel: S stages, x at the salient columns [16][s_pad] fp16, the rank-0
// CTA's slots for the other ranks' partial rows [C-1][256 threads][4 MT] floats, and barriers.
struct MbSmem {
  uint8_t* stages;
  __half* xs;
  float* slots;
  uint64_t* full;          // [S] stage landed
  uint64_t* empty;         // [S] consumers released the stage
  uint64_t* red_full;      // rank 0: every other rank wrote its partial rows of the tile
  uint64_t* red_empty;     // other ranks: rank 0 has read this rank's partial rows
  int* last_fill;          // [kMaxStagesMb]
};

template <int MT>  // n8 tiles of the batch: 1 for M <= 8, 2 for M <= 16
__global__ void __launch_bounds__(kMbThreads, 1)
    qtea_gemv_mb_kernel(const __grid_constant__ MbMaps maps, const __grid_constant__ MbParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int S = p.n_stages;
  const int C = p.cluster;                 // CTAs of a cluster share a tile, each a range of chunks
  const int rank = (int)cluster_rank();
  MbSmem sm;
  sm.stages = smem;
  sm.xs = reinterpret_cast<__half*>(smem + (size_t)S * kMbStageBytes);
  sm.slots = reinterpret_cast<float*>(smem + (size_t)S * kMbStageBytes + (size_t)16 * p.s_pad * 2);
  sm.full = reinterpret_cast<uint64_t*>(sm.slots + (size_t)(C - 1) * kMbConsumerWarps * 32 * 4 * MT);
  sm.empty = sm.full + S;
  sm.red_full = sm.empty + S;
  sm.red_empty = sm.red_full + 1;
  sm.last_fill = reinterpret_cast<int*>(sm.red_empty + 1);

  // tiles of this cluster: cluster_id, + n_clusters, ...; chunks of this CTA: [c0, c1)
  const int cid = (int)cluster_id(), ncl = (int)n_clusters();
  const int n_my_tiles = p.n_tiles > cid ? (p.n_tiles - 1 - cid) / ncl + 1 : 0;
  const int c0 = rank * p.n_chunks / C, c1 = (rank + 1) * p.n_chunks / C;
  const int my_chunks = c1 - c0;
  const int n_fills = n_my_tiles * my_chunks;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_u32(&sm.full[i]), 1);
      mbar_init(smem_u32(&sm.empty[i]), kMbConsumerWarps);
      sm.last_fill[i] = 0;
    }
    mbar_init(smem_u32(sm.red_full), (uint32_t)(C > 1 ? (C - 1) * kMbConsumerWarps * 32 : 1));  // unused if C == 1
    mbar_init(smem_u32(sm.red_empty), (uint32_t)(kMbConsumerWarps * 32));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == kMbConsumerWarps && lane < 3) {
    const CUtensorMap* m = lane == 0 ? &maps.codes : (lane == 1 ? &maps.x : &maps.v);
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
  }
  cluster_sync();  // barriers initialised in every CTA of the cluster before any remote arrival
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  if (warp == kMbConsumerWarps) {
    // ---------------------------------------------------------------- producer lane
    if (lane == 0) {
      for (int f = 0; f < n_fills; ++f) {
        const int st = f % S, ph = f / S;
        if (ph > 0 && !mbar_wait(smem_u32(&sm.empty[st]), (uint32_t)((ph - 1) & 1), p.status)) break;
        const int t = cid + (f / my_chunks) * ncl, ch = c0 + f % my_chunks;
        uint8_t* sb = sm.stages + (size_t)st * kMbStageBytes;
        const uint32_t bar = smem_u32(&sm.full[st]);
        mbar_arrive_expect_tx(bar, kMbCodeBytes + kMbXBytes + kMbVBytes);
        tma_load_2d(smem_u32(sb), &maps.codes, ch * kChunkRowBytes, t * kMbTileRows, bar);
#pragma unroll
        for (int j = 0; j < kChunkCols / kMbXBoxCols; ++j)
          tma_load_2d(smem_u32(sb + kMbCodeBytes + j * 2048), &maps.x, ch * kChunkCols + j * kMbXBoxCols, 0, bar);
        tma_load_2d(smem_u32(sb + kMbCodeBytes + kMbXBytes), &maps.v, ch * kChunkCols, 0, bar);
        tma_load_2d(smem_u32(sb + kMbCodeBytes + kMbXBytes + 512), &maps.v, ch * kChunkCols + 256, 0, bar);
        sm.last_fill[st] = ph + 1;
      }
    }
  } else {
    // ---------------------------------------------------------------- consumers
    // x at the salient columns, rows beyond M and columns beyond s zero
    for (int i = threadIdx.x; i < 16 * p.s_pad; i += kMbConsumerWarps * 32) {
      const int m = i / p.s_pad, c = i - m * p.s_pad;
      __half v = __float2half(0.f);
      if (m < p.M && c < p.s) {
        int col = __ldg(p.sal + c);
        col = col < 0 ? 0 : (col >= p.K ? p.K - 1 : col);
        v = __ushort_as_half(__ldg(p.x + (size_t)m * p.K + col));
      }
      sm.xs[i] = v;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kMbConsumerWarps * 32) : "memory");

    const int g = lane >> 2, q = lane & 3;
    const int r0 = warp * 16 + g;  // tile rows of the thread: r0 and r0 + 8
    const int tid = threadIdx.x;   // consumer index 0 .. 255
    int f = 0;
    bool ok = true;
    for (int ti = 0; ti < n_my_tiles && ok; ++ti) {
      const int t = cid + ti * ncl;
      const int row0 = t * kMbTileRows + r0, row1 = row0 + 8;
      const uint16_t al0 = row0 < p.N ? __ldg(p.alpha + row0) : (uint16_t)0;
      const uint16_t al1 = row1 < p.N ? __ldg(p.alpha + row1) : (uint16_t)0;
      float acc[MT][4], res[MT][4];
#pragma unroll
      for (int j = 0; j < MT; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][e] = res[j][e] = 0.f;

      for (int ch = c0; ch < c1; ++ch, ++f) {
        const int st = f % S;
        ok = mbar_wait(smem_u32(&sm.full[st]), (uint32_t)((f / S) & 1), p.status);
        if (!__all_sync(0xffffffffu, ok)) {
          ok = false;
          break;
        }
        const uint8_t* sb = sm.stages + (size_t)st * kMbStageBytes;
        const uint8_t* c0p = sb + (size_t)r0 * kChunkRowBytes;
        const uint8_t* c1p = c0p + 8 * kChunkRowBytes;
        const uint8_t* xb = sb + kMbCodeBytes;
        const uint32_t* vb = reinterpret_cast<const uint32_t*>(sb + kMbCodeBytes + kMbXBytes);
#pragma unroll 2
        for (int k4 = 0; k4 < 8; ++k4) {  // 16-byte chunk of codes = 4 steps of 16 columns
          const uint4 w0 = *reinterpret_cast<const uint4*>(c0p + ((k4 ^ (r0 & 7)) << 4));
          const uint4 w1 = *reinterpret_cast<const uint4*>(c1p + ((k4 ^ (r0 & 7)) << 4));
          const uint32_t wa[4] = {w0.x, w0.y, w0.z, w0.w};
          const uint32_t wb[4] = {w1.x, w1.y, w1.z, w1.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int kb = 4 * k4 + e;
            const uint2 vv = *reinterpret_cast<const uint2*>(vb + 8 * kb + 2 * q);  // v at 16kb + 4q .. +3
            uint32_t a0, a1, a2, a3;
            decode_byte(wa[e], (uint32_t)q, vv.x, vv.y, a0, a2);
            decode_byte(wb[e], (uint32_t)q, vv.x, vv.y, a1, a3);
            // x box kb / 4 holds columns 64 (kb / 4) .. +63; the step's 4q .. 4q+3 within it
            const int chunk = (kb & 3) * 2 + (q >> 1);
#pragma unroll
            for (int j = 0; j < MT; ++j) {
              const int n = 8 * j + g;
              const uint2 bb = *reinterpret_cast<const uint2*>(xb + (kb >> 2) * 2048 + n * 128 +
                                                               ((chunk ^ (n & 7)) << 4) + 8 * (q & 1));
              mma_16816(acc[j], a0, a1, a2, a3, bb.x, bb.y);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&sm.empty[st]));
      }
      if (!ok) break;

      // ---- residual (Eq. 11): virtual columns, 16 salient entries per step, steps split over ranks
      if (p.s > 0) {
        const int gq0 = row0 >> 2, gq1 = row1 >> 2, pos = row0 & 3;  // row1 & 3 == pos
        const bool v0 = gq0 < (p.N >> 2), v1 = gq1 < (p.N >> 2);
        const int rs = (p.s + 3) >> 2;
        for (int eb = rank; eb * 16 < p.s; eb += C) {
          const int e0 = eb * 16 + 4 * q;  // the thread's entries e0 .. e0 + 3
          uint2 r0v = make_uint2(0, 0), r1v = make_uint2(0, 0);
          uint32_t p0 = 0, p1 = 0;
          if (p.vec_res) {
            if (v0 && e0 < p.s) {
              r0v = __ldg(reinterpret_cast<const uint2*>(p.rvals + (size_t)gq0 * p.s + e0));
              p0 = __ldg(p.ridx + (size_t)gq0 * rs + (e0 >> 2));
            }
            if (v1 && e0 < p.s) {
              r1v = __ldg(reinterpret_cast<const uint2*>(p.rvals + (size_t)gq1 * p.s + e0));
              p1 = __ldg(p.ridx + (size_t)gq1 * rs + (e0 >> 2));
            }
          } else {
            uint32_t h0[4] = {0, 0, 0, 0}, h1[4] = {0, 0, 0, 0};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const int e = e0 + j;
              if (e < p.s) {
                if (v0) {
                  h0[j] = __ldg(p.rvals + (size_t)gq0 * p.s + e);
                  p0 |= ((uint32_t)(__ldg(p.ridx + (size_t)gq0 * rs + (e >> 2)) >> (2 * (e & 3))) & 3u) << (2 * j);
                }
                if (v1) {
                  h1[j] = __ldg(p.rvals + (size_t)gq1 * p.s + e);
                  p1 |= ((uint32_t)(__ldg(p.ridx + (size_t)gq1 * rs + (e >> 2)) >> (2 * (e & 3))) & 3u) << (2 * j);
                }
              }
            }
            r0v = make_uint2(h0[0] | (h0[1] << 16), h0[2] | (h0[3] << 16));
            r1v = make_uint2(h1[0] | (h1[1] << 16), h1[2] | (h1[3] << 16));
          }
          // keep the values whose stored position is this row (fp16 lanes all-ones or zero)
          auto keep = [&](uint32_t pb, int j0) -> uint32_t {
            const uint32_t lo = (((pb >> (2 * j0)) & 3u) == (uint32_t)pos) ? 0x0000ffffu : 0u;
            const uint32_t hi = (((pb >> (2 * j0 + 2)) & 3u) == (uint32_t)pos) ? 0xffff0000u : 0u;
            return lo | hi;
          };
          const uint32_t a0 = r0v.x & keep(p0, 0), a2 = r0v.y & keep(p0, 2);
          const uint32_t a1 = r1v.x & keep(p1, 0), a3 = r1v.y & keep(p1, 2);
#pragma unroll
          for (int j = 0; j < MT; ++j) {
            const int n = 8 * j + g;
            const uint2 bb = *reinterpret_cast<const uint2*>(sm.xs + (size_t)n * p.s_pad + e0);
            mma_16816(res[j], a0, a1, a2, a3, bb.x, bb.y);
          }
        }
      }

      // ---- this CTA's part of the tile: alpha * acc + res (alpha scales only the ternary part)
      const float fa0 = __half2float(__ushort_as_half(al0)), fa1 = __half2float(__ushort_as_half(al1));
      float part[MT][4];
#pragma unroll
      for (int j = 0; j < MT; ++j) {
        part[j][0] = fa0 * acc[j][0] + res[j][0];
        part[j][1] = fa0 * acc[j][1] + res[j][1];
        part[j][2] = fa1 * acc[j][2] + res[j][2];
        part[j][3] = fa1 * acc[j][3] + res[j][3];
      }
      if (rank != 0) {
        // into rank 0's slot for this rank, once rank 0 has read the previous tile's
        if (ti > 0 && !mbar_wait_cluster(smem_u32(sm.red_empty), (uint32_t)((ti - 1) & 1), p.status)) break;
        const uint32_t dst = map_rank(smem_u32(sm.slots + ((size_t)(rank - 1) * kMbConsumerWarps * 32 + tid) * 4 * MT), 0);
#pragma unroll
        for (int j = 0; j < MT; ++j) st_cluster_v4(dst + 16 * j, part[j][0], part[j][1], part[j][2], part[j][3]);
        mbar_arrive_cluster(map_rank(smem_u32(sm.red_full), 0));
        continue;
      }
      if (C > 1) {
        // rank 0: add the other ranks' parts in rank order, then give their slots back
        if (!mbar_wait_cluster(smem_u32(sm.red_full), (uint32_t)(ti & 1), p.status)) break;
        for (int rr = 1; rr < C; ++rr) {
          const float* src = sm.slots + ((size_t)(rr - 1) * kMbConsumerWarps * 32 + tid) * 4 * MT;
#pragma unroll
          for (int j = 0; j < MT; ++j) {
            const float4 v4 = *reinterpret_cast<const float4*>(src + 4 * j);
            part[j][0] += v4.x;
            part[j][1] += v4.y;
            part[j][2] += v4.z;
            part[j][3] += v4.w;
          }
        }
        for (int rr = 1; rr < C; ++rr) mbar_arrive_cluster(map_rank(smem_u32(sm.red_empty), (uint32_t)rr));
      }
      // ---- y[n][row] for the thread's rows and batch columns
#pragma unroll
      for (int j = 0; j < MT; ++j) {
        const int n0 = 8 * j + 2 * q;
        if (row0 < p.N) {
          if (n0 < p.M) p.y[(size_t)n0 * p.N + row0] = part[j][0];
          if (n0 + 1 < p.M) p.y[(size_t)(n0 + 1) * p.N + row0] = part[j][1];
        }
        if (row1 < p.N) {
          if (n0 < p.M) p.y[(size_t)n0 * p.N + row1] = part[j][2];
          if (n0 + 1 < p.M) p.y[(size_t)(n0 + 1) * p.N + row1] = part[j][3];
        }
      }
    }
  }

  // no bulk copy may still be writing shared memory when the CTA exits, and no CTA of the
  // cluster may exit while another may still write its shared memory
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int s2 = 0; s2 < S; ++s2) {
      const int lf = sm.last_fill[s2];
      if (lf > 0 && !mbar_wait(smem_u32(&sm.full[s2]), (uint32_t)((lf - 1) & 1), p.status)) break;
    }
  }
  cluster_sync();
}

}  // namespace

size_t mb_smem_bytes(int S, int s_pad, int cluster, int M) {
  const int mt = M <= 8 ? 1 : 2;
  return (size_t)S * kMbStageBytes + (size_t)16 * s_pad * 2 +
         (size_t)(cluster - 1) * kMbConsumerWarps * 32 * 4 * mt * sizeof(float) +
         (size_t)(2 * S + 2) * sizeof(unsigned long long) + (size_t)kMaxStagesMb * sizeof(int) + 1024;
}

cudaError_t mb_configure(size_t smem_optin, size_t* dyn_max) {
  cudaFuncAttributes a1, a2;
  cudaError_t e = cudaFuncGetAttributes(&a1, qtea_gemv_mb_kernel<1>);
  if (e != cudaSuccess) return e;
  e = cudaFuncGetAttributes(&a2, qtea_gemv_mb_kernel<2>);
  if (e != cudaSuccess) return e;
  const size_t st = a1.sharedSizeBytes > a2.sharedSizeBytes ? a1.sharedSizeBytes : a2.sharedSizeBytes;
  const size_t dyn = smem_optin > st ? smem_optin - st : 0;
  *dyn_max = dyn;
  e = cudaFuncSetAttribute(qtea_gemv_mb_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(qtea_gemv_mb_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
}

cudaError_t launch_mb(const MbMaps& maps, const MbParams& p, int grid, size_t smem, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kMbThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)p.cluster;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (p.M <= 8) return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<1>, maps, p);
  return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<2>, maps, p);
}

}  // namespace qtea
