// Row-resident batch-1 QTEA GEMV for sm_103a: y = alpha * (T . (v*x)) + sparse 1:4 residual, for
// groups of problems small enough that each CTA holds all the codes it needs at once.
//
// Computes Eq. 10 (one alpha per row, beta = 0) plus Eq. 11 of the QTEA paper (Sec. 3.5), with the
// same arithmetic as the stream-K batch-1 kernel (v*x staged per 512-column chunk as 16- or 24-bit
// fixed point in byte planes, dominant elements taken out and added exactly in fp32, codes
// multiplied with dp4a), but a decomposition built for latency rather than for streaming:
//  * Every CTA owns a block of whole rows (multiples of 8, at most 32: one per lane) of one problem,
//    so a row's sum is finished inside the CTA: no split-K workspace, no counters, no second CTA to
//    wait for. One CTA per SM where that covers the rows, else two. A wide launch (K above 4096, up
//    to 8192, or more than 256 salient columns) keeps one CTA per SM and its own instantiation.
//  * The CTA's codes arrive by TMA as 8-row x 128-byte boxes (128-byte swizzle) into one region per
//    512-column chunk, each region with its own barrier. The library owns the codes (no kernel
//    writes them after packing), so all of them are requested before griddepcontrol.wait, while
//    the preceding kernel on the stream still runs; the lines of x, v, the salient indices, the
//    CTA's residual rows and alpha are prefetched into L2 there too (a prefetch reads no value).
//  * After the wait, warp w takes chunks w, w + 8, ...: it stages the chunk's planes in its own
//    slot, waits for the chunk's codes and decodes them for all of the CTA's rows (each lane one
//    row with the stream-K kernel's decode loop; with 16 or 8 rows, two or four lanes per row,
//    each a part of the chunk). In a wide launch the next chunk's x and v are loaded before the
//    decode, so they arrive while it runs. Partial row sums meet in shared memory.
//  * The residual: each warp takes row groups of four, lanes over the salient entries, one sum
//    per position of the group. Its operands (values, positions, x at the salient columns) are
//    loaded right after the wait and held in registers across the decode, so their latency is
//    hidden behind it.
//  * y = alpha * sum + residual, written once per row, in a fixed order: results are bitwise
//    reproducible.
// The only wait is on the code barriers, bounded: after ~2 s the waiting warp records
// QTEA_ERR_TIMEOUT in the status word and stops; thread 0 drains the copies before the CTA exits.
#include <cuda_fp16.h>

#include "qtea_internal.h"
#include "qtea_m1_device.h"

namespace qtea {
namespace {

// Salient entries per lane held in registers: narrow launches 4 (the rest loaded in place), wide
// ones 16 (all of them).
template <bool WIDE>
__host__ __device__ constexpr int res_regs() { return WIDE ? kRowsMaxSalientWide / 32 : kRowsMaxSalient / 64; }
static_assert(kRowsMaxRows / 4 <= kRowsWarps, "one residual row group per warp");

// Decode one row (32 words of chunk-row bytes, 128-byte swizzle phase sw) against the chunk's P
// byte planes: the one-row form of decode_unit.
template <int P>
__device__ __forceinline__ void decode_row(const uint4* row0, const uint4* pl, int sw, RowAcc<P>& a0) {
  constexpr int kW = (P == 3) ? 3 : 2;
#pragma unroll
  for (int k = 0; k < P; ++k)
#pragma unroll
    for (int g = 0; g < 4; ++g) a0.a[k][g] = 0;
  uint4 P0 = pl[0], P1 = pl[1], P2 = kW == 3 ? pl[2] : make_uint4(0, 0, 0, 0);
  uint4 c0 = row0[0 ^ sw];
#pragma unroll 2
  for (int jj = 0; jj < 8; ++jj) {
    const uint4 n0 = row0[((jj + 1) & 7) ^ sw];
    const uint32_t w0[4] = {c0.x, c0.y, c0.z, c0.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int nw = ((4 * jj + e + 1) & 31) * 3;
      const uint4 Q0 = pl[nw], Q1 = pl[nw + 1];
      const uint4 Q2 = kW == 3 ? pl[nw + 2] : make_uint4(0, 0, 0, 0);
      if constexpr (P == 3) decode_word3(w0[e], P0, P1, P2, a0);
      else decode_word2(w0[e], P0, P1, a0);
      P0 = Q0;
      P1 = Q1;
      P2 = Q2;
    }
    c0 = n0;
  }
}

// T * v*x of the chunk's outliers for the row at byte base cb (swizzle phase sw).
__device__ __forceinline__ float outlier_sum(const ChunkMeta* mp, int n_out, const uint8_t* cb, int sw) {
  float o = 0.f;
#pragma unroll 1
  for (int k = 0; k < n_out; ++k) {
    const int col = mp->out_col[k];
    const int off = ((((col >> 6) ^ sw) << 4) | ((col >> 2) & 15)), sh = 2 * (col & 3);
    o = fmaf((float)(int)((cb[off] >> sh) & 3u) - 1.f, mp->out_val[k], o);
  }
  return o;
}

// Part k of kparts of one row's chunk (words k * W .. k * W + W - 1, W = 32 / kparts), taken in an
// order rotated by k so that the parts' plane reads fall in different banks. Each word is read with
// one 32-bit load from its 128-byte-swizzled granule; all W code words are loaded first, and each
// word's planes while the word before it decodes.
template <int P, int W>
__device__ __forceinline__ void decode_part(const uint8_t* row, const uint8_t* slot, int sw, int k, RowAcc<P>& a0) {
#pragma unroll
  for (int kk = 0; kk < P; ++kk)
#pragma unroll
    for (int g = 0; g < 4; ++g) a0.a[kk][g] = 0;
  auto word = [&](int t) { return k * W + ((t + k) & (W - 1)); };
  uint32_t code[W];
#pragma unroll
  for (int t = 0; t < W; ++t) {
    const int w = word(t);
    code[t] = *reinterpret_cast<const uint32_t*>(row + ((((w >> 2) ^ sw) << 4) | ((w & 3) << 2)));
  }
  const uint4* pw = reinterpret_cast<const uint4*>(slot + word(0) * kPlaneBytesPerWord);
  uint4 P0 = pw[0], P1 = pw[1], P2 = P == 3 ? pw[2] : make_uint4(0, 0, 0, 0);
#pragma unroll
  for (int t = 0; t < W; ++t) {
    uint4 Q0 = P0, Q1 = P1, Q2 = P2;
    if (t + 1 < W) {
      const uint4* qw = reinterpret_cast<const uint4*>(slot + word(t + 1) * kPlaneBytesPerWord);
      Q0 = qw[0];
      Q1 = qw[1];
      if constexpr (P == 3) Q2 = qw[2];
    }
    if constexpr (P == 3) decode_word3(code[t], P0, P1, P2, a0);
    else decode_word2(code[t], P0, P1, a0);
    P0 = Q0;
    P1 = Q1;
    P2 = Q2;
  }
}

// Chunk ch of the CTA's rows, with kparts lanes per row (row lane / kparts, part lane % kparts): the
// row's sum of T X scaled by q plus the outliers, added to part on every lane of the row. cs holds
// the chunk's fixed-point parameters as this warp staged them; the outlier list is in the slot.
template <int kparts>
__device__ __forceinline__ void decode_chunk(const uint8_t* region, const uint8_t* slot, int lane,
                                             const ChunkStage& cs, float& part) {
  const ChunkMeta* mp = reinterpret_cast<const ChunkMeta*>(slot + kAuxMeta);
  const float scale = cs.scale;
  const int planes = cs.planes, n_out = cs.n_out;
  const long long sum_x = cs.sum_x;
  const int row = kparts == 1 ? lane : lane / kparts, k = lane - row * kparts;
  const int sw = row & 7;  // 128-byte swizzle phase of the row
  const uint8_t* rb = region + (size_t)row * kChunkRowBytes;
  float d0;
  if constexpr (kparts == 1) {
    const uint4* pl = reinterpret_cast<const uint4*>(slot);
    if (planes == 2) {
      RowAcc<2> a0;
      decode_row<2>(reinterpret_cast<const uint4*>(rb), pl, sw, a0);
      d0 = finish_chunk2(a0, (int)sum_x);
    } else {
      RowAcc<3> a0;
      decode_row<3>(reinterpret_cast<const uint4*>(rb), pl, sw, a0);
      d0 = finish_chunk3(a0, sum_x);
    }
  } else {
    constexpr int W = 32 / kparts;
    if (planes == 2) {
      RowAcc<2> a0;
      decode_part<2, W>(rb, slot, sw, k, a0);
      d0 = finish_chunk2(a0, k == 0 ? (int)sum_x : 0);  // the chunk's sum of X once per row
    } else {
      RowAcc<3> a0;
      decode_part<3, W>(rb, slot, sw, k, a0);
      d0 = finish_chunk3(a0, k == 0 ? sum_x : 0ll);
    }
  }
  float v = d0 * scale;
  if (k == 0 && n_out > 0) v += outlier_sum(mp, n_out, rb, sw);
  for (int o = 1; o < kparts; o <<= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  part += v;
}

// Prefetch into L2 the bytes [p, p + n) (one prefetch per 128-byte line, lines t, t + T, ...).
__device__ __forceinline__ void prefetch_range(const void* p, size_t n, int t, int T) {
  if (!p || n == 0) return;
  const uintptr_t a = reinterpret_cast<uintptr_t>(p) & ~(uintptr_t)127;
  const uintptr_t e = reinterpret_cast<uintptr_t>(p) + n;
  for (uintptr_t l = a + (uintptr_t)t * 128; l < e; l += (uintptr_t)T * 128)
    asm volatile("prefetch.global.L2 [%0];" ::"l"(l) : "memory");
}

template <int KP, bool WIDE>
__global__ void __launch_bounds__(kRowsThreads, WIDE ? 1 : 2)
    qtea_gemv_rows_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ RowsParams rp) {
  constexpr int kResRegs = res_regs<WIDE>();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const RowsSmem so = rows_smem_layout(rp.rows_cap, rp.n_chunks_max);
  uint8_t* codes = smem;
  uint8_t* slot = smem + so.slots + (size_t)warp * kRowsSlotBytes;
  float* dec = reinterpret_cast<float*>(smem + so.dec);
  float* res = reinterpret_cast<float*>(smem + so.res);
  ProblemArgs* args = reinterpret_cast<ProblemArgs*>(smem + so.args);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + so.bars);

  // this CTA's problem and rows: 8-row blocks of the problem split evenly over its CTAs
  int p = 0;
  while (p + 1 < rp.n_problems && (int)blockIdx.x >= rp.cta_begin[p + 1]) ++p;
  const int ci = (int)blockIdx.x - rp.cta_begin[p], nc = rp.cta_begin[p + 1] - rp.cta_begin[p];
  if (tid < (int)(sizeof(ProblemArgs) / 4))
    reinterpret_cast<uint32_t*>(args)[tid] = reinterpret_cast<const uint32_t*>(&rp.prob[p])[tid];
  const int N = rp.prob[p].N, n_chunks = rp.prob[p].n_chunks;
  const int nb = (N + kRowsBoxRows - 1) / kRowsBoxRows;
  const int b0 = (int)((long long)nb * ci / nc), b1 = (int)((long long)nb * (ci + 1) / nc);
  const int r0 = b0 * kRowsBoxRows, r1 = min(b1 * kRowsBoxRows, N), R = r1 - r0;
  const int n_boxes = b1 - b0;
  if (warp == 0 && lane == 0)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.m[p])) : "memory");
  if (tid == 0) {
    for (int c = 0; c < n_chunks; ++c) mbar_init(smem_u32(&bars[c]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();

  // before the dependency wait: the codes (library-owned) and L2 prefetches of what the CTA reads
  if (warp == 0) {
    const CUtensorMap* map = &maps.m[p];
    for (int c = lane; c < n_chunks; c += 32) {
      const uint32_t bar = smem_u32(&bars[c]);
      const uint32_t dst = smem_u32(codes + (size_t)c * rp.rows_cap * kChunkRowBytes);
      mbar_arrive_expect_tx(bar, (uint32_t)(n_boxes * kRowsBoxRows * kChunkRowBytes));
      for (int j = 0; j < n_boxes; ++j)
        tma_load_2d(dst + (uint32_t)(j * kRowsBoxRows * kChunkRowBytes), map, c * kChunkRowBytes,
                    r0 + j * kRowsBoxRows, bar);
    }
  } else {
    const ProblemArgs& a = rp.prob[p];
    const int t = tid - 32, T = kRowsThreads - 32;
    prefetch_range(a.x, (size_t)a.K * 2, t, T);
    prefetch_range(a.v, (size_t)a.K * 2, t, T);
    prefetch_range(a.alpha + r0, (size_t)R * 2, t, T);
    if (a.s > 0) {
      const int rs = (a.s + 3) >> 2;
      prefetch_range(a.sal, (size_t)a.s * 4, t, T);
      prefetch_range(a.rvals + (size_t)(r0 / 4) * a.s, (size_t)(R / 4) * a.s * 2, t, T);
      prefetch_range(a.ridx + (size_t)(r0 / 4) * rs, (size_t)(R / 4) * rs, t, T);
    }
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  const ProblemArgs& a = *args;
  const int s = a.s;
  // lanes per row: 4 for up to 8 rows, 2 for 16, 1 for up to 32; KP > 0 when every CTA of the launch
  // takes the same (the variant then holds only that decode)
  const int kparts = KP ? KP : (R <= 8 ? 4 : R <= 16 ? 2 : 1);
  // the first chunk's x and v go out before everything else
  ChunkLoads L0;
  if (warp < n_chunks) load_chunk(a, warp, lane, L0);
  // loads whose values are needed last go out first: alpha of the thread's row; the residual
  // operands of the warp's row group (group `warp` of the CTA: R <= 32 rows make at most eight
  // groups; lane's entries lane + 32 i for i < kResRegs) and the salient columns, whose x goes out
  // once the first planes are staged
  const uint16_t al = tid < R ? __ldg(a.alpha + r0 + tid) : (uint16_t)0;
  const int rs = (s + 3) >> 2;
  const int q = r0 / 4 + warp;
  const bool has_group = s > 0 && warp < R / 4;
  uint32_t rv[kResRegs], pb[kResRegs];
  int col[kResRegs];
  uint32_t xsb[kResRegs];  // x at the salient columns, fp16 bits: converted only when the residual is formed
#pragma unroll
  for (int i = 0; i < kResRegs; ++i) {
    const int e = lane + 32 * i;
    const bool in = has_group && e < s;
    col[i] = in ? __ldg(a.sal + e) : 0;
    rv[i] = in ? __ldg(a.rvals + (size_t)q * s + e) : 0u;
    pb[i] = in ? __ldg(a.ridx + (size_t)q * rs + (e >> 2)) : 0u;
  }
  bool gathered = false;
  // x at the salient columns, in flight until the residual is formed (no instruction reads the
  // loaded registers before then, so the decode does not wait for them)
  auto gather = [&]() {
#pragma unroll
    for (int i = 0; i < kResRegs; ++i) {
      const int e = lane + 32 * i;
      const int cc = col[i] < 0 ? 0 : (col[i] >= a.K ? a.K - 1 : col[i]);
      xsb[i] = 0u;
      if (has_group && e < s) xsb[i] = __ldg(a.x + cc);
    }
    gathered = true;
  };

  float part = 0.f;
  bool ok = true;
  for (int c = warp; c < n_chunks; c += kRowsWarps) {
    ChunkStage cs;
    if (WIDE || c == warp) {
      cs = write_planes<false>(a, L0, slot, lane);
      // wide: the warp's next chunk's x and v go out now and arrive during this chunk's decode
      if (WIDE && c + kRowsWarps < n_chunks) load_chunk(a, c + kRowsWarps, lane, L0);
    } else {
      ChunkLoads L;
      load_chunk(a, c, lane, L);
      cs = write_planes<false>(a, L, slot, lane);
    }
    if (!gathered) gather();
    __syncwarp();
    ok = mbar_wait(smem_u32(&bars[c]), 0, rp.status);
    if (!__all_sync(0xffffffffu, ok)) {
      ok = false;
      break;
    }
    const uint8_t* region = codes + (size_t)c * rp.rows_cap * kChunkRowBytes;
    if (KP == 1 || (KP == 0 && kparts == 1)) decode_chunk<1>(region, slot, lane, cs, part);
    else if (KP == 2 || (KP == 0 && kparts == 2)) decode_chunk<2>(region, slot, lane, cs, part);
    else decode_chunk<4>(region, slot, lane, cs, part);
    __syncwarp();  // the slot is rewritten by the warp's next chunk
  }
  if (!gathered) gather();
  if (lane % kparts == 0)  // a timed-out warp: NaN rows
    dec[warp * kRowsMaxRows + lane / kparts] = ok ? part : __int_as_float(0x7fc00000);

  // the residual (Eq. 11) of the warp's row group: one sum per position of the group, lanes over
  // the salient entries (those past 32 * kResRegs loaded here), reduced across the warp
  if (has_group) {
    float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
#pragma unroll
    for (int i = 0; i < kResRegs; ++i) {
      const int e = lane + 32 * i;
      const float pr = h2f((uint16_t)rv[i]) * h2f((uint16_t)xsb[i]);  // zero past s
      const int pos = (pb[i] >> (2 * (e & 3))) & 3;
      acc0 += pos == 0 ? pr : 0.f;
      acc1 += pos == 1 ? pr : 0.f;
      acc2 += pos == 2 ? pr : 0.f;
      acc3 += pos == 3 ? pr : 0.f;
    }
#pragma unroll 1
    for (int e = lane + 32 * kResRegs; e < s; e += 32) {
      int cc = __ldg(a.sal + e);
      cc = cc < 0 ? 0 : (cc >= a.K ? a.K - 1 : cc);
      const float pr = h2f(__ldg(a.rvals + (size_t)q * s + e)) * h2f(__ldg(a.x + cc));
      const int pos = (__ldg(a.ridx + (size_t)q * rs + (e >> 2)) >> (2 * (e & 3))) & 3;
      acc0 += pos == 0 ? pr : 0.f;
      acc1 += pos == 1 ? pr : 0.f;
      acc2 += pos == 2 ? pr : 0.f;
      acc3 += pos == 3 ? pr : 0.f;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      acc0 += __shfl_xor_sync(0xffffffffu, acc0, o);
      acc1 += __shfl_xor_sync(0xffffffffu, acc1, o);
      acc2 += __shfl_xor_sync(0xffffffffu, acc2, o);
      acc3 += __shfl_xor_sync(0xffffffffu, acc3, o);
    }
    if (lane < 4) res[4 * warp + lane] = lane == 0 ? acc0 : lane == 1 ? acc1 : lane == 2 ? acc2 : acc3;
  }
  __syncthreads();

  if (tid < R) {
    float d = 0.f;
#pragma unroll
    for (int w = 0; w < kRowsWarps; ++w) d += dec[w * kRowsMaxRows + tid];
    const float r = s > 0 ? res[tid] : 0.f;
    a.y[r0 + tid] = fmaf(h2f(al), d, r);
  }
  // no bulk copy may still be writing shared memory when the CTA exits (after a timeout a warp
  // may not have waited for its chunks)
  if (tid == 0) {
    for (int c = 0; c < n_chunks; ++c)
      if (!mbar_wait(smem_u32(&bars[c]), 0, rp.status)) break;
  }
}

}  // namespace

cudaError_t rows_configure(size_t smem_optin) {
  for (auto k : {qtea_gemv_rows_kernel<0, false>, qtea_gemv_rows_kernel<1, false>, qtea_gemv_rows_kernel<2, false>,
                 qtea_gemv_rows_kernel<4, false>, qtea_gemv_rows_kernel<0, true>, qtea_gemv_rows_kernel<1, true>}) {
    const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_optin);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// Programmatic stream serialisation lets the launch start while the previous kernel on the
// stream drains.
cudaError_t launch_rows(const TensorMaps& maps, const RowsParams& p, int grid, size_t smem, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kRowsThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // lanes per row: a variant holding only that decode when every CTA takes the same; wide launches
  // (one CTA per SM) have a one-lane-per-row variant and the general one
  if (p.wide)
    return p.kparts == 1 ? cudaLaunchKernelEx(&cfg, qtea_gemv_rows_kernel<1, true>, maps, p)
                         : cudaLaunchKernelEx(&cfg, qtea_gemv_rows_kernel<0, true>, maps, p);
  return p.kparts == 4   ? cudaLaunchKernelEx(&cfg, qtea_gemv_rows_kernel<4, false>, maps, p)
         : p.kparts == 2 ? cudaLaunchKernelEx(&cfg, qtea_gemv_rows_kernel<2, false>, maps, p)
         : p.kparts == 1 ? cudaLaunchKernelEx(&cfg, qtea_gemv_rows_kernel<1, false>, maps, p)
                         : cudaLaunchKernelEx(&cfg, qtea_gemv_rows_kernel<0, false>, maps, p);
}

}  // namespace qtea
