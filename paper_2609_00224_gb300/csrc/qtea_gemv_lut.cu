// Batch-1 QTEA GEMV by table lookup, the decode the paper gives for its base-3 storage
// (Sec. 3.5; Appendix A): each code byte packs five ternary digits (3^5 = 243 < 256) and indexes a
// table of the dot products of those five columns' v*x with every digit pattern. The table is
// sign-symmetric: the pattern with every digit mirrored (code 242 - c) has the opposite value, and
// code 121 (five zeros) has value 0, so 122 entries per pack hold it: entry k = the value of code
// 121 + k, and code c < 121 reads entry 121 - c with the sign flipped (the half-LUT).
//
// Serves base-3 layouts at M = 1: one alpha per row, or the paper's storage with alpha and beta per
// row and group of 128 columns (Eq. 10), fp16 or FP8 residual values.
// Design for sm_103a:
//  * Work: a unit is (problem, 512-row tile, chunk of 8 blocks of 128 columns = 208 code bytes per
//    row). The units of all problems form one sequence split evenly over persistent CTAs (one per
//    SM); tiles split over CTAs are reduced as in the batch-1 dp4a kernel (partial rows in a
//    per-layout workspace, the last contributor summing them in CTA order: bitwise reproducible).
//  * Per unit the CTA builds the chunk's half-LUTs in shared memory: 208 packs x 122 fp32 entries,
//    each entry ((((t4 x4 + t3 x3) + t2 x2) + t1 x1) + t0 x0) in that fixed order (t = digit - 1,
//    x = v*x exact in fp32), so an entry's value does not depend on who builds it.
//  * Lookup: a warp takes 32 rows, 8 at a time. Lane l < 26 owns the chunk's code bytes 8l .. 8l+7
//    of every row (one 8-byte load per row); entry k of pack 8l + j sits at table column 26 j + l of
//    a 224-float table row, so the 26 lanes always read 26 distinct banks (no conflicts whatever the
//    codes). Per byte: |c - 121| -> shared load -> sign flip -> add. Each lane sums its 8 packs of
//    each row; two shuffle rounds and a transposed butterfly over the rest leave each of the 8 rows'
//    chunk sums in fixed lanes, in a fixed order.
//  * Scale groups of 128 columns: a lane's 8 packs lie in at most two blocks; their table values
//    are scaled by those blocks' alpha (staged with beta for the tile's rows and the chunk's blocks)
//    before the lanes are summed, and each row adds beta times the blocks' sums of x.
//  * Residual (Eq. 11): the chunk's share of the salient entries (blocks of 8 entries split over the
//    chunks by index, as in the dp4a kernel), x at their columns staged with the table; each lane
//    adds its row's entries (loads issued before the lookups, used after). Never scaled by alpha.
//  * No cross-CTA waiting, no mbarriers; caller memory is read after the grid dependency wait.
#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

// CTA whose range contains unit u.
__device__ __forceinline__ int unit_owner(long long u, long long total, int grid) {
  return (int)(((u + 1) * grid - 1) / total);
}

struct LutSmem {
  float* table;  // [kLutHalf][kLutStride]
  float* xt;     // [kLutCols] v*x of the chunk
  float* xs;     // [kLutMaxEntries] x at the salient columns of the chunk's entries
};

// Build the chunk's half-LUTs: warp w takes pack slot j = w % 8 of lanes l < 26 (pack 8l + j) and
// half (w / 8) of the 122 entries, walking the codes in order (lowest digit fastest) and keeping the
// partial sums of the higher digits.
__device__ __forceinline__ void build_table(const LutSmem& sm, int warp, int lane) {
  const int j = warp & 7, half = warp >> 3, l = lane;
  if (l >= kLutLanes) return;
  const int p = 8 * l + j;                    // pack = code byte of the chunk
  const int blk = p / 26, q = p - 26 * blk;  // block and byte within it
  float x[5];
#pragma unroll
  for (int d = 0; d < 5; ++d) {
    const int cb = 5 * q + d;                 // column within the block (pads past 127: x = 0)
    x[d] = cb < 128 ? sm.xt[blk * 128 + cb] : 0.f;
  }
  const int c0 = 121 + half * 61, c1 = half ? 243 : 182;
  int d0 = c0 % 3, d1 = (c0 / 3) % 3, d2 = (c0 / 9) % 3, d3 = (c0 / 27) % 3, d4 = c0 / 81;
  float s4 = (float)(d4 - 1) * x[4];
  float s3 = fmaf((float)(d3 - 1), x[3], s4);
  float s2 = fmaf((float)(d2 - 1), x[2], s3);
  float s1 = fmaf((float)(d1 - 1), x[1], s2);
  float* col = sm.table + 26 * j + l;
  for (int c = c0; c < c1; ++c) {
    col[(c - 121) * kLutStride] = fmaf((float)(d0 - 1), x[0], s1);
    if (++d0 == 3) {
      d0 = 0;
      if (++d1 == 3) {
        d1 = 0;
        if (++d2 == 3) {
          d2 = 0;
          if (++d3 == 3) {
            d3 = 0;
            ++d4;
            s4 = (float)(d4 - 1) * x[4];
          }
          s3 = fmaf((float)(d3 - 1), x[3], s4);
        }
        s2 = fmaf((float)(d2 - 1), x[2], s3);
      }
      s1 = fmaf((float)(d1 - 1), x[1], s2);
    }
  }
}

// Value of code byte c of table column base `colp` (pointer to entry 0 of the pack's column).
__device__ __forceinline__ float lookup(const float* colp, uint32_t c) {
  const int d = (int)c - 121;
  const float v = colp[(d < 0 ? -d : d) * kLutStride];
  return __int_as_float(__float_as_int(v) ^ (d & (int)0x80000000));
}

// Load the 8 code bytes of lane l for one row (bytes past the chunk's valid packs read as code
// 121, value 0).
__device__ __forceinline__ uint2 load_codes(const LutProblem& a, int row, int ch, int l, int valid_packs) {
  uint2 w = make_uint2(0x79797979u, 0x79797979u);
  if (row >= a.N || l >= kLutLanes) return w;
  const int b0 = 8 * l;
  const uint8_t* src = a.packed + (size_t)row * a.row_bytes + (size_t)ch * kLutPacks + b0;
  if (b0 + 8 <= valid_packs && a.aligned8) return __ldg(reinterpret_cast<const uint2*>(src));
  uint32_t byte[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) byte[k] = b0 + k < valid_packs ? (uint32_t)__ldg(src + k) : 0x79u;
  w.x = byte[0] | byte[1] << 8 | byte[2] << 16 | byte[3] << 24;
  w.y = byte[4] | byte[5] << 8 | byte[6] << 16 | byte[7] << 24;
  return w;
}

// The lane's 8 packs of one row (codes w): plain sum, or with scale groups each value times the
// alpha of its block (fa[j], the lo or hi block's alpha).
__device__ __forceinline__ float row_packs(const float* colp, uint2 w) {
  float s0 = 0.f, s1 = 0.f;
#pragma unroll
  for (int j = 0; j < 4; j += 2) {
    s0 += lookup(colp + 26 * j, (w.x >> (8 * j)) & 0xFFu);
    s1 += lookup(colp + 26 * (j + 1), (w.x >> (8 * (j + 1))) & 0xFFu);
  }
#pragma unroll
  for (int j = 0; j < 4; j += 2) {
    s0 += lookup(colp + 26 * (4 + j), (w.y >> (8 * j)) & 0xFFu);
    s1 += lookup(colp + 26 * (5 + j), (w.y >> (8 * (j + 1))) & 0xFFu);
  }
  return s0 + s1;
}

__device__ __forceinline__ float row_packs_grouped(const float* colp, uint2 w, int jb, float a_lo, float a_hi) {
  float s0 = 0.f, s1 = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t c = ((j < 4 ? w.x : w.y) >> (8 * (j & 3))) & 0xFFu;
    const float v = lookup(colp + 26 * j, c);
    if (j & 1) s1 = fmaf(j < jb ? a_lo : a_hi, v, s1);
    else s0 = fmaf(j < jb ? a_lo : a_hi, v, s0);
  }
  return s0 + s1;
}

// Sum of the 8 rows' values over the warp's 32 lanes: lanes l with l % 8 == r end with row r's sum.
__device__ __forceinline__ float reduce8(float (&v)[8], int lane) {
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], 16);
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], 8);
#pragma unroll
  for (int s = 4; s >= 1; s >>= 1) {
    const bool up = (lane & s) != 0;
#pragma unroll
    for (int i = 0; i < s; ++i) {
      const float send = up ? v[i] : v[i + s];
      const float keep = up ? v[i + s] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0];
}

template <bool GROUPED>
__global__ void __launch_bounds__(kLutThreads, 1) qtea_gemv_lut_kernel(const __grid_constant__ LutParams P) {
  extern __shared__ __align__(16) uint8_t smem[];
  LutSmem sm;
  sm.table = reinterpret_cast<float*>(smem);
  sm.xt = sm.table + kLutHalf * kLutStride;
  sm.xs = sm.xt + kLutCols;
  float* bsx = sm.xs + kLutMaxEntries;                                // [kLutBlocks] sums of x per block
  uint32_t* sab = reinterpret_cast<uint32_t*>(bsx + kLutBlocks);      // [kLutTileRows][kLutBlocks] (alpha, beta)
  // a lane's packs 8l .. 8l+7 lie in blocks b_lo and b_lo + 1; packs j < jb in b_lo
  const int b_lo = (8 * (threadIdx.x & 31)) / 26, jb = 26 * (b_lo + 1) - 8 * (threadIdx.x & 31);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int u0 = P.cta_u0[blockIdx.x], u1 = P.cta_u0[blockIdx.x + 1];
  const long long total = P.total_units;
  const int grid = gridDim.x;
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  int p = 0;
  while (p + 1 < P.n_problems && u0 >= P.prob[p + 1].unit_begin) ++p;
  float tacc = 0.f, racc = 0.f;  // this lane's row of the current tile: ternary sum, residual
  for (int u = u0; u < u1; ++u) {
    while (p + 1 < P.n_problems && u >= P.prob[p + 1].unit_begin) ++p;
    const LutProblem& a = P.prob[p];
    const int v = (int)(u - a.unit_begin), t = v / a.n_chunks, ch = v - t * a.n_chunks;
    const int nbk = min(kLutBlocks, a.n_blocks - ch * kLutBlocks);  // blocks in this chunk
    // the chunk's salient entries: blocks of 8 entries split over the chunks by index
    const int nb = (a.s + 7) / 8;
    const int e0 = (int)((long long)ch * nb / a.n_chunks) * 8;
    const int e1 = min((int)((long long)(ch + 1) * nb / a.n_chunks) * 8, a.s);
    const int row = t * kLutTileRows + warp * 32 + lane;
    const int qg = row >> 2, pos = row & 3;

    // the first 8 rows' codes go out before the table is built (their latency overlaps it)
    const int valid_packs = 26 * nbk;
    const int rbase = t * kLutTileRows + warp * 32;
    uint2 cw[8], nw[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) cw[r] = load_codes(a, rbase + r, ch, lane, valid_packs);

    __syncthreads();  // the previous unit's table is no longer read
    for (int i = threadIdx.x; i < kLutCols; i += kLutThreads) {
      const int col = ch * kLutCols + i;
      sm.xt[i] = col < a.K ? h2f(__ldg(a.v + col)) * h2f(__ldg(a.x + col)) : 0.f;  // exact in fp32
    }
    if (GROUPED) {
      // alpha and beta (0 without the bias option) of the tile's rows and the chunk's blocks, and the
      // blocks' sums of x (in column order, by one warp per block)
      for (int i = threadIdx.x; i < kLutTileRows * kLutBlocks; i += kLutThreads) {
        const int r = i / kLutBlocks, b = i - r * kLutBlocks, rg = t * kLutTileRows + r;
        const int g = (ch * kLutBlocks + b) / a.gdiv;  // the block's scale group
        uint32_t ab = 0;
        if (rg < a.N && b < nbk) {
          const uint16_t* sc = a.scales + (size_t)rg * a.G * (a.bias ? 2 : 1) + (size_t)g * (a.bias ? 2 : 1);
          ab = (uint32_t)__ldg(sc) | (a.bias ? (uint32_t)__ldg(sc + 1) << 16 : 0u);
        }
        sab[i] = ab;
      }
      if (warp < kLutBlocks) {
        float sx = 0.f;
        for (int c = lane; c < 128; c += 32) {
          const int col = ch * kLutCols + warp * 128 + c;
          sx += col < a.K ? h2f(__ldg(a.x + col)) : 0.f;
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) sx += __shfl_xor_sync(0xffffffffu, sx, o);
        if (lane == 0) bsx[warp] = sx;
      }
    }
    for (int e = e0 + threadIdx.x; e < e1; e += kLutThreads) {
      int col = __ldg(a.sal + e);
      col = col < 0 ? 0 : (col >= a.K ? a.K - 1 : col);
      sm.xs[e - e0] = h2f(__ldg(a.x + col));
    }
    __syncthreads();
    build_table(sm, warp, lane);
    __syncthreads();

    // residual of this lane's row over the chunk's entries: loads go out before the lookups
    float res = 0.f;
    const bool row_ok = row < a.N;
    uint32_t rvw[kLutResBatch / 2];  // values, two per word (fp16 bits, or an FP8 byte in each half)
    uint32_t rpw[kLutResBatch / 16];  // positions, sixteen 2-bit fields per word
    const int rs = (a.s + 3) >> 2;
    auto load_res = [&](int eb) {
      const int n = row_ok ? min(kLutResBatch, e1 - eb) : 0;
#pragma unroll
      for (int k = 0; k < kLutResBatch / 2; ++k) rvw[k] = 0;
#pragma unroll
      for (int k = 0; k < kLutResBatch / 16; ++k) rpw[k] = 0;
#pragma unroll
      for (int k = 0; k < kLutResBatch; ++k) {
        if (k < n) {
          const size_t e = (size_t)qg * a.s + eb + k;
          const uint32_t val = a.fp8 ? (uint32_t)__ldg(reinterpret_cast<const uint8_t*>(a.rvals) + e)
                                     : (uint32_t)__ldg(reinterpret_cast<const uint16_t*>(a.rvals) + e);
          rvw[k >> 1] |= val << (16 * (k & 1));
          const int ee = eb + k;
          const uint32_t pb = __ldg(a.ridx + (size_t)qg * rs + (ee >> 2));
          rpw[k >> 4] |= ((pb >> (2 * (ee & 3))) & 3u) << (2 * (k & 15));
        }
      }
    };
    if (e1 > e0) load_res(e0);

    // lookups: 32 rows of the warp, 8 rows per batch, the next batch's codes loaded ahead
    const float* colp = sm.table + lane;  // + 26 j + k * kLutStride
    float chunk_sum = 0.f;                // row `row` over the chunk (alpha applied with scale groups)
#pragma unroll 1
    for (int bt = 0; bt < 4; ++bt) {
      if (bt < 3) {
#pragma unroll
        for (int r = 0; r < 8; ++r) nw[r] = load_codes(a, rbase + 8 * (bt + 1) + r, ch, lane, valid_packs);
      }
      float acc[8];
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        if (lane >= kLutLanes) {
          acc[r] = 0.f;
        } else if (GROUPED) {
          const uint32_t* ab = sab + (warp * 32 + 8 * bt + r) * kLutBlocks;
          const float a_lo = h2f((uint16_t)(ab[b_lo] & 0xFFFFu));
          const float a_hi = jb < 8 ? h2f((uint16_t)(ab[b_lo + 1] & 0xFFFFu)) : 0.f;
          acc[r] = row_packs_grouped(colp, cw[r], jb, a_lo, a_hi);
        } else {
          acc[r] = row_packs(colp, cw[r]);
        }
      }
      const float s8 = reduce8(acc, lane);  // row rbase + 8 bt + lane % 8
      if ((lane >> 3) == bt) chunk_sum = s8;
#pragma unroll
      for (int r = 0; r < 8; ++r) cw[r] = nw[r];
    }
    if (GROUPED) {  // beta times the blocks' sums of x
      const uint32_t* ab = sab + (warp * 32 + lane) * kLutBlocks;
#pragma unroll
      for (int b = 0; b < kLutBlocks; ++b) chunk_sum = fmaf(h2f((uint16_t)(ab[b] >> 16)), bsx[b], chunk_sum);
    }

    for (int eb = e0; eb < e1; eb += kLutResBatch) {
      if (eb > e0) load_res(eb);
      const int n = min(kLutResBatch, e1 - eb);
#pragma unroll
      for (int k = 0; k < kLutResBatch; ++k) {
        const uint32_t pk = (rpw[k >> 4] >> (2 * (k & 15))) & 3u;
        if (k < n && (int)pk == pos) {  // entries past n hold position 0 and value 0
          const uint32_t bits = (rvw[k >> 1] >> (16 * (k & 1))) & 0xFFFFu;
          const float r = a.fp8 ? e4m3_to_float(bits) : h2f((uint16_t)bits);
          res = fmaf(r, sm.xs[eb - e0 + k], res);
        }
      }
    }
    tacc += chunk_sum;
    racc += res;

    // tile epilogue once this CTA's part of tile t is done
    if (ch == a.n_chunks - 1 || u == u1 - 1) {
      const long long A = a.unit_begin + (long long)t * a.n_chunks, B = A + a.n_chunks;
      const float al = GROUPED ? 1.f : (row_ok ? h2f(__ldg(a.scales + row)) : 0.f);
      const float val = fmaf(al, tacc, racc);
      const int tr = warp * 32 + lane;  // row within the tile
      if (A >= u0 && B <= u1) {
        if (row_ok) a.y[row] = val;
      } else {
        const int my_slot = (u0 >= A) ? 0 : 1;
        a.ws[((size_t)blockIdx.x * 2 + my_slot) * kLutTileRows + tr] = val;
        __syncwarp();
        const int bf = unit_owner(A, total, grid), bl = unit_owner(B - 1, total, grid);
        int last = 0;
        if (lane == 0) {
          unsigned* ctr = a.counters + (size_t)t * kLutWarps + warp;
          unsigned prev;
          asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], 1;" : "=r"(prev) : "l"(ctr) : "memory");
          last = (prev == (unsigned)(bl - bf));
          if (last) *ctr = 0u;
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          float s = 0.f;
          for (int cb = bf; cb <= bl; ++cb) {
            const int cslot = (P.cta_u0[cb] >= A) ? 0 : 1;
            s += __ldcg(a.ws + ((size_t)cb * 2 + cslot) * kLutTileRows + tr);
          }
          if (row_ok) a.y[row] = s;
        }
      }
      tacc = racc = 0.f;
    }
  }
}

}  // namespace

cudaError_t lut_configure(size_t smem_optin) {
  if (kLutSmemBytes > smem_optin) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(qtea_gemv_lut_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kLutSmemBytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(qtea_gemv_lut_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kLutSmemBytes);
}

cudaError_t launch_lut(const LutParams& p, bool grouped, int grid, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kLutThreads);
  cfg.dynamicSmemBytes = kLutSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return grouped ? cudaLaunchKernelEx(&cfg, qtea_gemv_lut_kernel<true>, p)
                 : cudaLaunchKernelEx(&cfg, qtea_gemv_lut_kernel<false>, p);
}

}  // namespace qtea
