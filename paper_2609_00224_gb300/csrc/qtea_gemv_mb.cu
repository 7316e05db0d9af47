// Tensor-core QTEA GEMV for sm_103a: y[m] = x[m] * W^T for 2 <= M <= 16 batch rows, and for
// 2-bit layouts in the paper's storage at any M.
//
// Computes Eq. 10 (one alpha per row, or alpha and beta per row and 128-column group) plus Eq. 11
// of the QTEA paper (Sec. 3.5). With M rows the product is a skinny dense contraction, so it runs on
// mma.sync m16n8k16 (fp16 operands, fp32 accumulation), exactly:
//  * A = 2T * v. A 32-bit code word holds the codes c = T + 1 of 16 consecutive columns; shifting
//    it left by 14 - 2i puts the codes of columns i and i + 8 at bits 14-15 and 30-31, and one
//    LOP3 (~w & 0xC000C000) turns each into the fp16 value -2, -0 or +2 (sign bit and the top
//    exponent bit). One multiply by the pair (v_i, v_{i+8}) gives 2T * v exactly (a power-of-two
//    multiple of an fp16 value). The accumulator is halved once (per group with scale groups).
//  * B = x, the fp16 activations, unchanged; each product is exact in fp32 and the sums
//    accumulate in fp32. The contraction index runs over the columns in the order that pairing
//    gives (columns i and i + 8 of a word side by side), so v and x of each 512-column chunk are
//    written once per call in exactly the register order the fragments need ("fragment order"):
//    one 8-byte shared load per thread and step. Each MMA step stays inside one 128-column group.
//  * Split encoding, M <= 4: v moves into B, so A = 2T needs only the shift and the mask. B holds
//    v*x * 2^E (exact in fp32, E per chunk so that every value stays below 2^15) as two fp16
//    columns per batch row, hi = fp16(v*x 2^E) and lo = fp16(v*x 2^E - hi), whose sum is exact;
//    the tile's chunks are folded one by one with their 2^(-E-1). Rows whose code is 0 at a column
//    contribute 0 there, as with 2T*v (an encoding by c = T + 1 would carry a large activation
//    into every row's accumulator and lose the others' low bits to its alignment).
//  * The residual of Eq. 11 is an exact contraction too: over "virtual columns", one per salient
//    column, A holds the residual value (fp16, or FP8 E4M3 converted exactly) of the row's group
//    where the stored position is the row and 0 elsewhere, and B holds x at the salient column.
//    Helper warps compute it per 256-row tile from bulk-copied residual rows, off the decode's
//    path; it is added, unscaled by alpha, at the tile's end.
// Work: a unit is 256 rows x 512 columns of one problem; the units of every problem of a group form
// one sequence split evenly over persistent CTAs (one cooperative launch for all the GEMVs of a
// group). The consumer threads first build the fragment-order chunks (spread over the CTAs; each
// CTA's own first chunk straight into its first stage), then decode. Each of eight consumer warps
// owns two 16-row blocks of a unit, so every B fragment it loads feeds two MMAs; two accumulator
// sets alternate between steps. A tile whose units span several CTAs is finished by the CTA holding
// its first unit, which reaches it at the end of its range; the others store their partial rows
// (self-validating words) and carry on without waiting. The sum runs in CTA order, so results do
// not depend on timing. A producer lane streams the CTA's units through a ring of
// shared-memory stages: 256 rows x 128 bytes of codes by TMA (128-byte swizzle), the chunk's v and
// x in fragment order by bulk copy, and with scale groups the unit's alpha (and beta) by TMA.
// |v| must stay below 32768 (2v is formed in fp16). Every wait is bounded (~2 s, then
// QTEA_ERR_TIMEOUT in the status word).
#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

constexpr int kMbThreads = (kMbConsumerWarps + 1 + kMbHelperWarps) * 32;  // consumers, producer, helpers
constexpr int kMbCodeBytes = kMbTileRows * kChunkRowBytes;  // 32768

// 1-D bulk copy of `bytes` (a multiple of 16, both addresses 16-byte aligned) into shared memory.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
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

// Codes of columns I and I + 8 of word w as fp16 -2, -0 or +2 (2T), times the pair of v.
template <int I>
__device__ __forceinline__ uint32_t a_reg(uint32_t w, uint32_t vpair) {
  const uint32_t t2 = ~(w << (14 - 2 * I)) & 0xC000C000u;
  return h2_as_u32(__hmul2(u32_as_h2(t2), u32_as_h2(vpair)));
}

// Partial rows of split tiles are stored XOR-ed with this NaN bit pattern, so that zeroed memory
// reads as "not written yet" and every 4-byte word validates itself (no result has this pattern).
constexpr uint32_t kPartEmpty = 0x7FBADBADu;

// Loads and stores of those words are strong (relaxed, GPU scope): a weak load may keep returning a
// stale copy of the line (the two dies' L2 partitions), so it need not ever see another CTA's store.
__device__ __forceinline__ uint4 part_load4(const uint4* p) {
  uint4 w;
  asm volatile("ld.relaxed.gpu.global.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(w.x), "=r"(w.y), "=r"(w.z), "=r"(w.w)
               : "l"(p)
               : "memory");
  return w;
}
__device__ __forceinline__ void part_store4(uint4* p, uint4 w) {
  asm volatile("st.relaxed.gpu.global.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(w.x), "r"(w.y), "r"(w.z), "r"(w.w)
               : "memory");
}
__device__ __forceinline__ bool part_written4(const uint4& w) { return w.x && w.y && w.z && w.w; }

// CTA whose range contains unit u (the inverse of the balanced split cta_u0[b] = b * total / grid).
__device__ __forceinline__ int unit_owner(long long u, long long total, int grid) {
  return (int)(((u + 1) * grid - 1) / total);
}

struct UnitPos {
  int p, t, ch;  // problem, tile, chunk
};

__device__ __forceinline__ UnitPos unit_pos(const MbProblemArgs* tab, int n_problems, long long u) {
  int p = 0;
  while (p + 1 < n_problems && u >= tab[p + 1].unit_begin) ++p;
  const int v = (int)(u - tab[p].unit_begin);
  const int nc = tab[p].n_chunks;
  const int t = v / nc;
  return {p, t, v - t * nc};
}

// ---------------------------------------------------------------- prep kernel

// Residual (Eq. 11) of one 16-entry step for a consumer thread's rows: the values whose stored
// position is the row (fp16 lanes all-ones or zero) as A, x at the salient columns as B. Entries
// e0 .. e0 + 3 (e0 = 16 step + 4q) of the row groups of rows r, r + 8 of block b (r = tr + 16b + g)
// come from the staged tile: rv [64 groups][rvs] fp16, ri [64][ris] position bytes (entry e of a
// group in bits 2(e % 4) of byte e / 4), xr [16 batch rows][xrs] fp16 (zero past the valid
// entries); only entries below ne count.
// FP8 E4M3 (bias 7, subnormals m * 2^-9, NaN at S.1111.111, no infinity) as fp16 bits; every value
// is exactly representable in fp16.
__device__ __forceinline__ uint32_t e4m3_to_f16_bits(uint32_t b) {
  const uint32_t e = (b >> 3) & 15u, m = b & 7u;
  uint32_t mag;
  if (e == 0u) mag = __half_as_ushort(__float2half_rn((float)m * 0.001953125f));  // m * 2^-9, exact
  else if (e == 15u && m == 7u) mag = 0x7e00u;
  else mag = ((e + 8u) << 10) | (m << 7);
  return ((b & 0x80u) << 8) | mag;
}

// FP8: rv holds one E4M3 byte per entry (row stride rvs bytes), converted to fp16 exactly.
// With the split encoding (split) B column n of tile j holds batch row 4j + n/2 for even n and zero
// for odd n, so that the result sits where the decode's (hi, lo) pair of that batch row does.
template <int NB, bool FP8 = false>
__device__ __forceinline__ void res_step(const void* rv_, int rvs, const uint8_t* ri, int ris, const uint16_t* xr,
                                         int xrs, int ne, int step, int tr, int g, int q, int mt, bool split,
                                         bool quad_loads, float (&res)[NB][2][4]) {
  const uint16_t* rv = static_cast<const uint16_t*>(rv_);
  const uint8_t* rv8 = static_cast<const uint8_t*>(rv_);
  const int e0 = step * 16 + 4 * q;
  const uint32_t pos = (uint32_t)(g & 3);  // row & 3 for every row of the thread
  uint2 xb[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    if (split) xb[j] = (g & 1) ? make_uint2(0u, 0u) : *reinterpret_cast<const uint2*>(xr + (4 * j + (g >> 1)) * xrs + e0);
    else xb[j] = *reinterpret_cast<const uint2*>(xr + (8 * j + g) * xrs + e0);
  }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    uint32_t a[4];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int gl = (tr + 16 * b + 8 * h + g) >> 2;
      // match bits: field k of d is zero where entry e0 + k is stored at this row's position;
      // nz holds bit 2k set where it is not
      const uint32_t d = (uint32_t)ri[gl * ris + (e0 >> 2)] ^ (pos * 0x55u);
      const uint32_t nz = (d | (d >> 1)) & 0x55u;
      uint32_t lo, hi;
      if (FP8) {
        uint32_t q4 = 0;  // the four E4M3 bytes
        if (quad_loads) {  // one 4-byte load (rvs % 4 == 0)
          if (e0 < ne) q4 = *reinterpret_cast<const uint32_t*>(rv8 + gl * rvs + e0);
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k) q4 |= (e0 + k < ne ? (uint32_t)rv8[gl * rvs + e0 + k] : 0u) << (8 * k);
        }
        lo = e4m3_to_f16_bits(q4 & 0xffu) | (e4m3_to_f16_bits((q4 >> 8) & 0xffu) << 16);
        hi = e4m3_to_f16_bits((q4 >> 16) & 0xffu) | (e4m3_to_f16_bits(q4 >> 24) << 16);
      } else if (quad_loads) {  // the four values in one 8-byte load (rvs % 4 == 0, e0 + 3 < ne or zero)
        uint2 v = make_uint2(0, 0);
        if (e0 < ne) v = *reinterpret_cast<const uint2*>(rv + gl * rvs + e0);
        lo = v.x;
        hi = v.y;
      } else {
        uint32_t v4[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) v4[k] = e0 + k < ne ? (uint32_t)rv[gl * rvs + e0 + k] : 0u;
        lo = v4[0] | (v4[1] << 16);
        hi = v4[2] | (v4[3] << 16);
      }
      // keep a 16-bit lane where its match bit is clear: (bit - 1) is all ones exactly then
      const uint32_t k0 = ((nz & 1u) - 1u) & 0x0000ffffu, k1 = (((nz >> 2) & 1u) - 1u) & 0xffff0000u;
      const uint32_t k2 = (((nz >> 4) & 1u) - 1u) & 0x0000ffffu, k3 = (((nz >> 6) & 1u) - 1u) & 0xffff0000u;
      a[h] = lo & (k0 | k1);
      a[2 + h] = hi & (k2 | k3);
    }
    mma_16816(res[b][0], a[0], a[1], a[2], a[3], xb[0].x, xb[0].y);
    if (mt == 2) mma_16816(res[b][1], a[0], a[1], a[2], a[3], xb[1].x, xb[1].y);
  }
}

// v and x of chunk ch of problem p in fragment order, and the group sums of x, to out (global
// memory or a stage): 256 threads (tid), sm holds 17,408 bytes of scratch, sync() is a barrier over
// the 256 threads. Entry (step s, quad
// lane q) of the v block holds the pairs (v[16W + i], v[16W + i + 8]) for i = 2(s & 3) and i + 1,
// W = 4(s >> 2) + q; entry (step s, lane 4g + q) of x block j holds the same two pairs of x[8j + g].
// Columns >= K and batch rows >= M are zero. Steps 8k .. 8k + 7 cover columns 128k .. 128k + 127.
template <typename Sync>
__device__ __forceinline__ void prep_chunk(const MbPrepProblem& p, int M, int mt, int ch, int tid, uint8_t* sm,
                                           uint8_t* out, Sync sync) {
  uint16_t(*xsm)[kChunkCols] = reinterpret_cast<uint16_t(*)[kChunkCols]>(sm);
  uint16_t* vsm = reinterpret_cast<uint16_t*>(sm + 16 * kChunkCols * 2);
  const int col0 = ch * kChunkCols;
#pragma unroll 2
  for (int i = tid; i < kChunkCols; i += 256) {
    const int col = col0 + i;
    const bool in = col < p.K;
    vsm[i] = in ? __ldg(p.v + col) : (uint16_t)0;
    uint16_t xv[16];
#pragma unroll
    for (int m = 0; m < 16; ++m) xv[m] = (in && m < M) ? __ldg(p.x + (size_t)m * p.K + col) : (uint16_t)0;
#pragma unroll
    for (int m = 0; m < 16; ++m) xsm[m][i] = xv[m];
  }
  sync();
  auto pair = [](const uint16_t* row, int c) { return (uint32_t)row[c] | ((uint32_t)row[c + 8] << 16); };
  if (tid < 128) {
    const int s = tid >> 2, q = tid & 3;
    const int base = 16 * (4 * (s >> 2) + q), i0 = 2 * (s & 3);
    reinterpret_cast<uint2*>(out)[tid] = make_uint2(pair(vsm, base + i0), pair(vsm, base + i0 + 1));
  }
  for (int e = tid; e < mt * 1024; e += 256) {
    const int j = e >> 10, s = (e >> 5) & 31, lane = e & 31, g = lane >> 2, q = lane & 3;
    const int base = 16 * (4 * (s >> 2) + q), i0 = 2 * (s & 3);
    const uint16_t* row = xsm[8 * j + g];
    reinterpret_cast<uint2*>(out + kMbChunkHead)[e] = make_uint2(pair(row, base + i0), pair(row, base + i0 + 1));
  }
  {
    // sum of x over each 128-column group k of the chunk for batch row m (the beta term of Eq. 10):
    // four lanes per (k, m) add 32 columns each, then a fixed butterfly
    const int k = tid >> 6, m = (tid >> 2) & 15, part = tid & 3;
    float sxv = 0.f;
#pragma unroll 8
    for (int c = 0; c < 32; ++c) sxv += __half2float(__ushort_as_half(xsm[m][128 * k + 32 * part + c]));
    sxv += __shfl_xor_sync(0xffffffffu, sxv, 1);
    sxv += __shfl_xor_sync(0xffffffffu, sxv, 2);
    if (part == 0) reinterpret_cast<float*>(out + kMbVBytes)[16 * k + m] = sxv;
  }
}

// Largest of the lanes' non-negative values (their bit patterns order as unsigned integers).
__device__ __forceinline__ float warp_max_nonneg(float v) {
  return __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(v)));
}

// The split encoding's chunk (M <= 8): B = the exact fp16 split hi + lo of v*x * 2^E, with
// E = 14 - floor(log2(max |v*x|)) over the chunk and all batch rows (every |v*x * 2^E| < 2^15, so
// hi is finite; v*x is exact in fp32 and hi + lo holds all of its bits); in tile j, B column n is
// hi (n even) or lo (n odd) of batch row 4j + n/2, zero for batch rows >= M. A is 2T (split_a), so
// the head holds the fold factor 2^(-E-1) and, as for the other encoding, the sums of x per
// 128-column group and batch row (the beta term). 256 threads (tid); sm holds kMbPrepScratch bytes;
// sync() is a barrier over the 256 threads.
template <typename Sync>
__device__ __forceinline__ void prep_chunk_split(const MbPrepProblem& p, int M, int mt, int ch, int tid, uint8_t* sm,
                                                 uint8_t* out, Sync sync) {
  uint16_t(*xsm)[kChunkCols] = reinterpret_cast<uint16_t(*)[kChunkCols]>(sm);
  uint16_t* vsm = reinterpret_cast<uint16_t*>(sm + 16 * kChunkCols * 2);
  float* red = reinterpret_cast<float*>(sm + 16 * kChunkCols * 2 + kChunkCols * 2);  // [8] warp maxima
  const int col0 = ch * kChunkCols;
  float lmax = 0.f;
#pragma unroll 2
  for (int i = tid; i < kChunkCols; i += 256) {
    const int col = col0 + i;
    const bool in = col < p.K;
    const uint16_t vb = in ? __ldg(p.v + col) : (uint16_t)0;
    vsm[i] = vb;
    const float vf = h2f(vb);
    uint16_t xv[16];
#pragma unroll
    for (int m = 0; m < 16; ++m) xv[m] = (in && m < M) ? __ldg(p.x + (size_t)m * p.K + col) : (uint16_t)0;
#pragma unroll
    for (int m = 0; m < 16; ++m) {
      xsm[m][i] = xv[m];
      lmax = fmaxf(lmax, fabsf(vf * h2f(xv[m])));
    }
  }
  lmax = warp_max_nonneg(lmax);
  if ((tid & 31) == 0) red[tid >> 5] = lmax;
  sync();
  float amax = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) amax = fmaxf(amax, red[w]);
  // |v*x| >= 2^-48 when nonzero (products of binary16 values), so amax is an fp32 normal number
  const int e = amax > 0.f ? (int)((__float_as_uint(amax) >> 23) & 0xffu) - 127 : 0;
  const float sc = __uint_as_float((uint32_t)(141 - e) << 23);  // 2^E, E = 14 - e
  auto half_of = [&](const uint16_t* row, int c, int h) -> uint32_t {
    const float f = (h2f(vsm[c]) * h2f(row[c])) * sc;  // exact: a power-of-two multiple of v*x
    const __half hi = __float2half_rn(f);
    if (h == 0) return (uint32_t)__half_as_ushort(hi);
    return (uint32_t)__half_as_ushort(__float2half_rn(f - __half2float(hi)));
  };
  for (int idx = tid; idx < mt * 1024; idx += 256) {
    const int j = idx >> 10, st = (idx >> 5) & 31, lane = idx & 31, g = lane >> 2, q = lane & 3;
    const int m = 4 * j + (g >> 1), h = g & 1;
    const int c0 = 16 * (4 * (st >> 2) + q) + 2 * (st & 3), c1 = c0 + 1;
    uint2 o = make_uint2(0u, 0u);
    if (m < M) {
      o.x = half_of(xsm[m], c0, h) | (half_of(xsm[m], c0 + 8, h) << 16);
      o.y = half_of(xsm[m], c1, h) | (half_of(xsm[m], c1 + 8, h) << 16);
    }
    reinterpret_cast<uint2*>(out + kMbChunkHead)[idx] = o;
  }
  {
    // sum of x over each 128-column group k of the chunk for batch row m (the beta term of Eq. 10):
    // four lanes per (k, m) add 32 columns each, then a fixed butterfly
    const int k = tid >> 6, m = (tid >> 2) & 15, part = tid & 3;
    float sxv = 0.f;
#pragma unroll 8
    for (int c = 0; c < 32; ++c) sxv += h2f(xsm[m][128 * k + 32 * part + c]);
    sxv += __shfl_xor_sync(0xffffffffu, sxv, 1);
    sxv += __shfl_xor_sync(0xffffffffu, sxv, 2);
    if (part == 0) reinterpret_cast<float*>(out + kMbVBytes)[16 * k + m] = sxv;
    if (tid == 0) *reinterpret_cast<float*>(out + kMbHlF) = __uint_as_float((uint32_t)(112 + e) << 23);  // 2^(-E-1)
  }
}

// x at salient columns 256 blk .. 256 blk + 255 of problem p, all 16 batch rows (xs[m][c], zero
// beyond s or M); one column per thread.
__device__ __forceinline__ void prep_gather(const MbPrepProblem& p, int M, int blk, int tid) {
  const int c = blk * 256 + tid;
  if (c < p.s16) {
    int col = c < p.s ? __ldg(p.sal + c) : 0;
    col = col < 0 ? 0 : (col >= p.K ? p.K - 1 : col);
    uint16_t xv[16];
#pragma unroll
    for (int m = 0; m < 16; ++m) xv[m] = (c < p.s && m < M) ? __ldg(p.x + (size_t)m * p.K + col) : (uint16_t)0;
#pragma unroll
    for (int m = 0; m < 16; ++m) p.xs[(size_t)m * p.s16 + c] = xv[m];
  }
}

// Blocks of a problem: its chunks; then, for a residual left to the prep kernel, its 256-row tiles;
// or, for a residual of the main kernel's helpers, blocks that gather x at the salient columns
// (xs[m][c], zero beyond s or M), 256 columns each.
// Tile t: the residual of its 256 rows for every batch row, computed with the main kernel's thread
// mapping (thread tid holds rows tr + 16b + g and + 8, batch rows 8j + 2q and + 1) and stored in
// that order, so that each main-kernel thread reads its part with vector loads. The tile's values
// and position bytes are one contiguous range each, starting on a 16-byte boundary (64 groups x s
// x 2 bytes and 64 groups x ceil(s/4) bytes before it); with `native` they are copied as they are
// by 16-byte loads, otherwise (too large for shared memory, or not 16-byte aligned) in passes of
// kMbResEntries entries by 2-byte loads.
__global__ void __launch_bounds__(256) qtea_mb_prep_kernel(const __grid_constant__ MbPrepGroup gr) {
  static_assert(kMbConsumerWarps * 32 == 256, "the prep kernel's residual blocks mirror the consumers");
  extern __shared__ __align__(16) uint8_t sm[];
  // the main kernel may launch now and prefetch its codes; it reads this kernel's output only after
  // its own grid dependency wait, which waits for this grid to complete
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  int pi = 0;
  while (pi + 1 < gr.n_problems && (int)blockIdx.x >= gr.prob[pi + 1].block_begin) ++pi;
  // the problem's fields in registers, read once (field-by-field reads from the parameter space
  // with a dynamic index would each be a constant-cache miss)
  const MbPrepProblem p = gr.prob[pi];
  const int M = gr.M;
  const int local = (int)blockIdx.x - p.block_begin;
  const int tid = threadIdx.x;
  if (local >= p.n_chunks && p.res_mode == kMbResHelpers) {
    prep_gather(p, M, local - p.n_chunks, tid);
    return;
  }
  if (local >= p.n_chunks) {
    // ---- residual of tile t
    const int t = local - p.n_chunks;
    const int g0 = t * (kMbTileRows / 4), ng = min(kMbTileRows / 4, p.N / 4 - g0);
    const int rs = (p.s + 3) >> 2;
    const int warp = tid >> 5, lane = tid & 31, g = lane >> 2, q = lane & 3;
    const int tr = warp * 16 * kMbBlocks;
    float res[kMbBlocks][2][4];
#pragma unroll
    for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
      for (int j = 0; j < 2; ++j)
#pragma unroll
        for (int k = 0; k < 4; ++k) res[b][j][k] = 0.f;
    const int E = p.native ? p.s : kMbResEntries;       // entries per pass
    const int xrs = (E + 15) & ~15;                       // staged x row stride
    const int ris = p.native ? rs : kMbResEntries / 4;  // staged position-byte row stride
    uint16_t* rv = reinterpret_cast<uint16_t*>(sm);
    uint8_t* ri = sm + (((size_t)64 * E * 2 + 15) & ~(size_t)15);
    uint16_t* xr = reinterpret_cast<uint16_t*>(ri + (((size_t)64 * ris + 15) & ~(size_t)15));
    for (int e_base = 0; e_base < p.s; e_base += E) {
      const int ne = min(E, p.s - e_base);
      if (p.native) {
        // whole 16-byte vectors by vector loads (all in flight at once), the tails by 2-byte and
        // 1-byte loads: no load past the caller's arrays
        const uint4* src = reinterpret_cast<const uint4*>(p.rvals + (size_t)g0 * p.s);
        uint4* dst = reinterpret_cast<uint4*>(rv);
        const int nv = (ng * p.s) >> 3;
#pragma unroll 16
        for (int i = tid; i < nv; i += 256) dst[i] = __ldg(src + i);
        for (int i = 8 * nv + tid; i < ng * p.s; i += 256) rv[i] = __ldg(p.rvals + (size_t)g0 * p.s + i);
        const uint4* srci = reinterpret_cast<const uint4*>(p.ridx + (size_t)g0 * rs);
        uint4* dsti = reinterpret_cast<uint4*>(ri);
        const int nvi = (ng * rs) >> 4;
#pragma unroll 4
        for (int i = tid; i < nvi; i += 256) dsti[i] = __ldg(srci + i);
        for (int i = 16 * nvi + tid; i < ng * rs; i += 256) ri[i] = __ldg(p.ridx + (size_t)g0 * rs + i);
      } else {
#pragma unroll 8
        for (int i = tid; i < 64 * kMbResEntries; i += 256) {
          const int gg = i / kMbResEntries, e = i % kMbResEntries;
          rv[i] = (gg < ng && e < ne) ? __ldg(p.rvals + (size_t)(g0 + gg) * p.s + e_base + e) : (uint16_t)0;
        }
#pragma unroll 8
        for (int i = tid; i < 64 * (kMbResEntries / 4); i += 256) {
          const int gg = i / (kMbResEntries / 4), e4 = i % (kMbResEntries / 4);
          ri[i] = (gg < ng && 4 * e4 < ne) ? __ldg(p.ridx + (size_t)(g0 + gg) * rs + (e_base >> 2) + e4) : (uint8_t)0;
        }
      }
      // x at the pass's salient columns (zero past ne): up to four entries per thread, their
      // column indices first, then all their x loads at once
      for (int e_lo = 0; e_lo < xrs; e_lo += 1024) {
        int col[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int e = e_lo + tid + 256 * k;
          col[k] = e < ne ? __ldg(p.sal + e_base + e) : 0;
          col[k] = col[k] < 0 ? 0 : (col[k] >= p.K ? p.K - 1 : col[k]);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int e = e_lo + tid + 256 * k;
          if (e >= xrs) break;
          uint16_t xv[16];
#pragma unroll
          for (int m = 0; m < 16; ++m) xv[m] = (m < M && e < ne) ? __ldg(p.x + (size_t)m * p.K + col[k]) : (uint16_t)0;
#pragma unroll
          for (int m = 0; m < 16; ++m) xr[m * xrs + e] = xv[m];
        }
      }
      __syncthreads();
      // groups past ng are never read: their rows lie past N, which the main kernel does not write
      const int rvs = p.native ? p.s : kMbResEntries;
      // 8-byte value loads where a row's entries start on 8-byte boundaries and the last quad is
      // whole (staged rows in passes are padded with zeros)
      const bool quad = (rvs & 3) == 0 && (p.native ? (ne & 3) == 0 : true);
      if (quad) {
        for (int step = 0; step * 16 < ne; ++step)
          res_step<kMbBlocks>(rv, rvs, ri, ris, xr, xrs, ne, step, tr, g, q, gr.mt, gr.split != 0, true, res);
      } else {
        for (int step = 0; step * 16 < ne; ++step)
          res_step<kMbBlocks>(rv, rvs, ri, ris, xr, xrs, ne, step, tr, g, q, gr.mt, gr.split != 0, false, res);
      }
      __syncthreads();
    }
    float4* dst = reinterpret_cast<float4*>(p.yres + ((size_t)t * 256 + tid) * 4 * kMbBlocks * gr.mt);
#pragma unroll
    for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
      for (int j = 0; j < 2; ++j)
        if (j < gr.mt) dst[b * gr.mt + j] = make_float4(res[b][j][0], res[b][j][1], res[b][j][2], res[b][j][3]);
    return;
  }
  if (gr.split)
    prep_chunk_split(p, M, gr.mt, local, tid, sm, p.ws + (size_t)local * kMbChunkWsBytes, [] { __syncthreads(); });
  else
    prep_chunk(p, M, gr.mt, local, tid, sm, p.ws + (size_t)local * kMbChunkWsBytes, [] { __syncthreads(); });
}

// ---------------------------------------------------------------- decode of one unit

// Group k of the unit done: run += alpha_k * (acc[0] + acc[1]) / 2 + beta_k * sum_k(x), acc = 0.
// alpha and beta of row r come from the unit's scale block (8 fp16 per row: (alpha, beta) of groups
// 0 .. 3 with beta, else alpha of groups 0 .. 7 of the chunk pair), the group sums from the chunk.
template <int MT>
__device__ __forceinline__ void group_fold(const uint8_t* sb, int tr, int g, int q, int k, int ch_odd, bool bias,
                                           float (&acc)[2][kMbBlocks][MT][4], float (&run)[kMbBlocks][MT][4]) {
  const uint16_t* ab = reinterpret_cast<const uint16_t*>(sb + kMbCodeBytes + kMbChunkHead + MT * kMbXTileBytes);
  const float* sx = reinterpret_cast<const float*>(sb + kMbCodeBytes + kMbVBytes) + 16 * k;
  float2 sxm[MT];
#pragma unroll
  for (int j = 0; j < MT; ++j) sxm[j] = *reinterpret_cast<const float2*>(sx + 8 * j + 2 * q);
#pragma unroll
  for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint16_t* r = ab + (tr + 16 * b + 8 * h + g) * 8;
      const float al = 0.5f * __half2float(__ushort_as_half(bias ? r[2 * k] : r[4 * ch_odd + k]));
      const float be = bias ? __half2float(__ushort_as_half(r[2 * k + 1])) : 0.f;
#pragma unroll
      for (int j = 0; j < MT; ++j) {
        run[b][j][2 * h] += al * (acc[0][b][j][2 * h] + acc[1][b][j][2 * h]) + be * sxm[j].x;
        run[b][j][2 * h + 1] += al * (acc[0][b][j][2 * h + 1] + acc[1][b][j][2 * h + 1]) + be * sxm[j].y;
        acc[0][b][j][2 * h] = acc[1][b][j][2 * h] = 0.f;
        acc[0][b][j][2 * h + 1] = acc[1][b][j][2 * h + 1] = 0.f;
      }
    }
}

// Split encoding: the accumulated steps of 128-column group k (or of the whole chunk, k < 0, without
// scale groups) folded into run: for batch row m = 4j + q, sum_j T v x = (D_hi + D_lo) * 2^(-E-1)
// (A = 2T, B = v*x 2^E); with scale groups times alpha_k plus beta_k times the group's sum of x
// (Eq. 10 per group). Only run[.][.][0] (row g) and [2] (row g + 8) carry values. acc = 0 afterwards.
template <int MT, bool GRP>
__device__ __forceinline__ void split_fold(const uint8_t* sb, int tr, int g, int q, int k, int ch_odd, bool bias,
                                           float (&acc)[2][kMbBlocks][MT][4], float (&run)[kMbBlocks][MT][4]) {
  const uint8_t* head = sb + kMbCodeBytes;
  const float F = *reinterpret_cast<const float*>(head + kMbHlF);
  const float* sx = reinterpret_cast<const float*>(head + kMbVBytes);
  const uint16_t* ab = reinterpret_cast<const uint16_t*>(sb + kMbCodeBytes + kMbChunkHead + MT * kMbXTileBytes);
#pragma unroll
  for (int j = 0; j < MT; ++j) {
    const float bx = GRP ? sx[16 * k + 4 * j + q] : 0.f;
#pragma unroll
    for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const float d = (acc[0][b][j][2 * h] + acc[0][b][j][2 * h + 1]) + (acc[1][b][j][2 * h] + acc[1][b][j][2 * h + 1]);
        if (GRP) {
          const uint16_t* r = ab + (tr + 16 * b + 8 * h + g) * 8;
          const float al = __half2float(__ushort_as_half(bias ? r[2 * k] : r[4 * ch_odd + k]));
          const float be = bias ? __half2float(__ushort_as_half(r[2 * k + 1])) : 0.f;
          run[b][j][2 * h] += fmaf(al * F, d, be * bx);
        } else {
          run[b][j][2 * h] = fmaf(d, F, run[b][j][2 * h]);
        }
        acc[0][b][j][2 * h] = acc[1][b][j][2 * h] = 0.f;
        acc[0][b][j][2 * h + 1] = acc[1][b][j][2 * h + 1] = 0.f;
      }
  }
}

// Split encoding, A = 2T of columns I and I + 8 of code word w: a left shift by 14 - 2I puts their
// codes c = T + 1 at bits 14-15 and 30-31, and one LOP3 (~w & 0xC000C000) turns each into the fp16
// value -2, -0 or +2 (sign bit and the top exponent bit). The shift is written as a multiply, which
// may issue on the multiply pipe beside the masks.
template <int I>
__device__ __forceinline__ uint32_t split_a(uint32_t w) {
  uint32_t t;
  asm("mul.lo.u32 %0, %1, %2;" : "=r"(t) : "r"(w), "n"(1u << (14 - 2 * I)));
  return ~t & 0xC000C000u;
}

// The unit's 32 steps of 16 columns for the warp's 16-row blocks (rows tr + 16b + g and + 8 of the
// stage); even steps accumulate into acc[0], odd steps into acc[1]. With scale groups (GRP) the
// steps of each 128-column group k (8k .. 8k + 7) are folded into run after the group's last step:
// run += alpha_k * acc / 2 + beta_k * sum_k(x), acc = 0 (Eq. 10 per group). With the split encoding
// (SPLIT) A is 2T (split_a) and B the chunk's (hi, lo) of v*x; without scale groups the unit's steps
// are folded into run at its end (split_fold).
template <int MT, bool GRP, bool SPLIT>
__device__ __forceinline__ void decode_unit(const uint8_t* sb, int tr, int g, int q, int lane, int ch_odd, bool bias,
                                            float (&acc)[2][kMbBlocks][MT][4], float (&run)[kMbBlocks][MT][4]) {
  const uint8_t* vblk = sb + kMbCodeBytes;
  const uint8_t* xblk = vblk + kMbChunkHead;
  // the thread's code words 4w + q (w = 0 .. 7) of each of its rows: word 4w + q sits in 16-byte
  // segment w of the row, stored at segment w ^ (row & 7) (128-byte swizzle); the 32 lanes of a load
  // hit 32 different banks
  uint32_t wr[kMbBlocks][2][8];
#pragma unroll
  for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint8_t* rp = sb + (size_t)(tr + 16 * b + 8 * h + g) * kChunkRowBytes + 4 * q;
#pragma unroll
      for (int w = 0; w < 8; ++w) wr[b][h][w] = *reinterpret_cast<const uint32_t*>(rp + ((w ^ g) << 4));
    }
  if constexpr (SPLIT) {
#pragma unroll
    for (int w = 0; w < 8; ++w) {
#pragma unroll
      for (int tq = 0; tq < 4; ++tq) {
        const int s = 4 * w + tq;
        uint32_t a[kMbBlocks][4];
#pragma unroll
        for (int b = 0; b < kMbBlocks; ++b) {
          if (tq == 0) {
            a[b][0] = split_a<0>(wr[b][0][w]); a[b][1] = split_a<0>(wr[b][1][w]);
            a[b][2] = split_a<1>(wr[b][0][w]); a[b][3] = split_a<1>(wr[b][1][w]);
          } else if (tq == 1) {
            a[b][0] = split_a<2>(wr[b][0][w]); a[b][1] = split_a<2>(wr[b][1][w]);
            a[b][2] = split_a<3>(wr[b][0][w]); a[b][3] = split_a<3>(wr[b][1][w]);
          } else if (tq == 2) {
            a[b][0] = split_a<4>(wr[b][0][w]); a[b][1] = split_a<4>(wr[b][1][w]);
            a[b][2] = split_a<5>(wr[b][0][w]); a[b][3] = split_a<5>(wr[b][1][w]);
          } else {
            a[b][0] = split_a<6>(wr[b][0][w]); a[b][1] = split_a<6>(wr[b][1][w]);
            a[b][2] = split_a<7>(wr[b][0][w]); a[b][3] = split_a<7>(wr[b][1][w]);
          }
        }
#pragma unroll
        for (int j = 0; j < MT; ++j) {
          const uint2 bx = *reinterpret_cast<const uint2*>(xblk + j * kMbXTileBytes + (s * 32 + lane) * 8);
#pragma unroll
          for (int b = 0; b < kMbBlocks; ++b)
            mma_16816(acc[s & 1][b][j], a[b][0], a[b][1], a[b][2], a[b][3], bx.x, bx.y);
        }
        if (GRP && (w & 1) && tq == 3) split_fold<MT, GRP>(sb, tr, g, q, w >> 1, ch_odd, bias, acc, run);
      }
    }
    if (!GRP) split_fold<MT, GRP>(sb, tr, g, q, -1, ch_odd, bias, acc, run);
    return;
  }
#pragma unroll
  for (int w = 0; w < 8; ++w) {
#pragma unroll
    for (int tq = 0; tq < 4; ++tq) {
      const int s = 4 * w + tq;
      const uint2 vp = *reinterpret_cast<const uint2*>(vblk + (s * 4 + q) * 8);
      // k slots 2q, 2q+1: columns i, i + 8 with i = 2tq; slots 2q+8, 2q+9: i = 2tq + 1
      uint32_t a[kMbBlocks][4];
#pragma unroll
      for (int b = 0; b < kMbBlocks; ++b) {
        if (tq == 0) {
          a[b][0] = a_reg<0>(wr[b][0][w], vp.x); a[b][1] = a_reg<0>(wr[b][1][w], vp.x);
          a[b][2] = a_reg<1>(wr[b][0][w], vp.y); a[b][3] = a_reg<1>(wr[b][1][w], vp.y);
        } else if (tq == 1) {
          a[b][0] = a_reg<2>(wr[b][0][w], vp.x); a[b][1] = a_reg<2>(wr[b][1][w], vp.x);
          a[b][2] = a_reg<3>(wr[b][0][w], vp.y); a[b][3] = a_reg<3>(wr[b][1][w], vp.y);
        } else if (tq == 2) {
          a[b][0] = a_reg<4>(wr[b][0][w], vp.x); a[b][1] = a_reg<4>(wr[b][1][w], vp.x);
          a[b][2] = a_reg<5>(wr[b][0][w], vp.y); a[b][3] = a_reg<5>(wr[b][1][w], vp.y);
        } else {
          a[b][0] = a_reg<6>(wr[b][0][w], vp.x); a[b][1] = a_reg<6>(wr[b][1][w], vp.x);
          a[b][2] = a_reg<7>(wr[b][0][w], vp.y); a[b][3] = a_reg<7>(wr[b][1][w], vp.y);
        }
      }
#pragma unroll
      for (int j = 0; j < MT; ++j) {
        const uint2 bx = *reinterpret_cast<const uint2*>(xblk + j * kMbXTileBytes + (s * 32 + lane) * 8);
#pragma unroll
        for (int b = 0; b < kMbBlocks; ++b) mma_16816(acc[s & 1][b][j], a[b][0], a[b][1], a[b][2], a[b][3], bx.x, bx.y);
      }
      if (GRP && (w & 1) && tq == 3) group_fold<MT>(sb, tr, g, q, w >> 1, ch_odd, bias, acc, run);
    }
  }
}

// ---------------------------------------------------------------- helper warps (residual)

__device__ __forceinline__ void helpers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kMbHelperWarps * 32) : "memory"); }
__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 2, %0;" ::"n"(kMbConsumerWarps * 32) : "memory");
}

// Arrival at the grid-wide barrier of a cooperative launch: one thread adds one to a monotonic
// counter, release at GPU scope (after a barrier over the threads whose writes it publishes).
__device__ __forceinline__ void grid_arrive(unsigned long long* bar) {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
  asm volatile("red.release.gpu.global.add.u64 [%0], 1;" ::"l"(bar) : "memory");
}

// One thread waits until every CTA arrived (acquire at GPU scope); bounded, a timeout is recorded in
// the status word. Data the other CTAs wrote is then read by bulk copies (async proxy).
__device__ __forceinline__ void grid_wait(const unsigned long long* bar, unsigned long long target, int* status) {
  const unsigned long long t0 = global_ns();
  for (;;) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(bar) : "memory");
    if (v >= target) break;
    if (global_ns() - t0 > kWaitLimitNs) {
      atomicExch(status, (int)QTEA_ERR_TIMEOUT);
      break;
    }
  }
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// The residual (Eq. 11) of every tile whose first chunk this CTA decodes, in the order the consumers
// reach those tiles, into a ring of two result slots laid out in the consumers' accumulator order
// ([256 consumer threads][4 kMbBlocks MT] floats). Per tile, in 1, 2 or 4 passes over its row
// groups: the pass's values and position bytes (one contiguous range each, starting on a 16-byte
// boundary) and, once per tile, x at the salient columns come by bulk copy (the last < 16 bytes by
// plain loads); then helper warp hw takes 16-row blocks hw, hw + 4, ... of the pass with the same
// virtual-column MMA as the prep kernel. A wait that times out is recorded in the status word and
// the helpers carry on, so that every helper reaches every named barrier.
template <int MT, bool SPLIT>
__device__ __noinline__ void helper_role(const MbProblemArgs* tab, int NP, int u0, int n_units, float* rslot,
                                         uint8_t* rstage, uint64_t* res_full, uint64_t* res_empty, uint64_t* staged,
                                         const MbGroupParams& gp, int hw, int lane, int* status) {
  const int g = lane >> 2, q = lane & 3;
  const int htid = hw * 32 + lane;
  // x at the salient columns is gathered by the CTAs before the grid barrier (with fused prep work)
  if (gp.fused) grid_wait(gp.gbar, gp.gbar_target, status);
  asm volatile("fence.proxy.async.global;" ::: "memory");
  UnitPos c = unit_pos(tab, NP, u0);
  int k = 0, sphase = 0;
  bool failed = false;
  for (int i = 0; i < n_units; ++i) {
    const MbProblemArgs& a = tab[c.p];
    if (c.ch == 0 && a.res_mode == kMbResHelpers) {
      const int slot = k & 1;
      const int s = a.s, rs = (s + 3) >> 2, s16 = a.s16;
      const int passes = a.res_passes, gpp = (kMbTileRows / 4) / passes;
      const int g0 = c.t * (kMbTileRows / 4), ng_tile = min(kMbTileRows / 4, a.N / 4 - g0);
      const int es = a.fp8 ? 1 : 2;  // bytes per residual value
      uint8_t* rv = rstage;
      uint8_t* ri = rstage + (((size_t)gpp * s * es + 15) & ~(size_t)15);
      uint16_t* xr = reinterpret_cast<uint16_t*>(ri + (((size_t)gpp * rs + 15) & ~(size_t)15));
      float* out = rslot + (size_t)slot * 256 * 8 * MT;
      if (k >= 2 && !mbar_wait(smem_u32(&res_empty[slot]), (uint32_t)(((k >> 1) - 1) & 1), status)) failed = true;
      const bool quad = (s & 3) == 0;
      for (int pass = 0; pass < passes; ++pass) {
        const int G0 = pass * gpp;
        const int ng = max(0, min(gpp, ng_tile - G0));
        helpers_sync();  // every helper is done with the staging buffer
        const size_t vb = (size_t)ng * s * es, ib = (size_t)ng * rs;
        const size_t vsrc = (size_t)(g0 + G0) * s * es, isrc = (size_t)(g0 + G0) * rs;  // bytes
        const uint8_t* rvals = reinterpret_cast<const uint8_t*>(a.rvals);
        if (htid == 0) {
          const uint32_t vbb = (uint32_t)(vb & ~(size_t)15), ibb = (uint32_t)(ib & ~(size_t)15);
          const uint32_t xbb = pass == 0 ? (uint32_t)(32 * s16) : 0u;
          const uint32_t bar = smem_u32(staged);
          // the helpers' reads of the previous pass (generic proxy) before the copies (async proxy)
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          mbar_arrive_expect_tx(bar, vbb + ibb + xbb);
          if (vbb) bulk_load(smem_u32(rv), rvals + vsrc, vbb, bar);
          if (ibb) bulk_load(smem_u32(ri), a.ridx + isrc, ibb, bar);
          if (xbb) bulk_load(smem_u32(xr), a.xs, xbb, bar);
        }
        {
          const int vt = (int)(vb & 15), it = (int)(ib & 15);  // tail bytes
          const size_t v0 = vb & ~(size_t)15, i0 = ib & ~(size_t)15;
          if (htid < vt) rv[v0 + htid] = __ldg(rvals + vsrc + v0 + htid);
          if (htid >= 32 && htid - 32 < it) ri[i0 + htid - 32] = __ldg(a.ridx + isrc + i0 + htid - 32);
        }
        if (!mbar_wait(smem_u32(staged), (uint32_t)(sphase & 1), status)) failed = true;
        ++sphase;
        helpers_sync();  // the tails are visible to every helper
        if (ng == 0) continue;  // rows past N: never written
        for (int jb = 0; jb < gpp / 16; ++jb) {
          const int rb = G0 / 4 + hw + 4 * jb;  // 16-row block of the tile
          float res[1][2][4];
#pragma unroll
          for (int j = 0; j < 2; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) res[0][j][e] = 0.f;
          const int tr = 16 * (rb - G0 / 4);  // first row of the block within the pass
          if (a.fp8) {
            for (int step = 0; step * 16 < s; ++step)
              res_step<1, true>(rv, s, ri, rs, xr, s16, s, step, tr, g, q, MT, SPLIT, quad, res);
          } else if (quad) {
            for (int step = 0; step * 16 < s; ++step) res_step<1>(rv, s, ri, rs, xr, s16, s, step, tr, g, q, MT, SPLIT, true, res);
          } else {
            for (int step = 0; step * 16 < s; ++step) res_step<1>(rv, s, ri, rs, xr, s16, s, step, tr, g, q, MT, SPLIT, false, res);
          }
          // consumer thread 32 (rb / 2) + lane holds these rows as its block rb % 2
          float4* dst = reinterpret_cast<float4*>(out + (size_t)(32 * (rb >> 1) + lane) * 8 * MT);
#pragma unroll
          for (int j = 0; j < MT; ++j) dst[(rb & 1) * MT + j] = make_float4(res[0][j][0], res[0][j][1], res[0][j][2], res[0][j][3]);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&res_full[slot]));
      ++k;
    }
    if (++c.ch == a.n_chunks) {
      c.ch = 0;
      if (++c.t == a.n_tiles) {
        c.t = 0;
        ++c.p;
      }
    }
  }
  // no bulk copy may still be writing shared memory when the CTA exits
  if (failed && htid == 0 && sphase > 0) mbar_wait(smem_u32(staged), (uint32_t)((sphase - 1) & 1), status);
}

// ---------------------------------------------------------------- main kernel

// MT: n8 tiles of the B operand (mb_mt). GRP: alpha (and beta) per row and 128-column group, loaded
// per unit by TMA, instead of one alpha per row. SPLIT: the split encoding (mb_split), else 2T * v.
template <int MT, bool GRP, bool SPLIT>
__global__ void __launch_bounds__(kMbThreads, 1)
    qtea_gemv_mb_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ TensorMaps ab_maps,
                        const __grid_constant__ MbGroupParams gp) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  constexpr int kStage = mb_stage_bytes(MT, GRP);
  constexpr uint32_t kFill = kMbCodeBytes + kMbChunkHead + MT * kMbXTileBytes + (GRP ? kMbAbBytes : 0);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int S = gp.n_stages;
  const int NP = gp.n_problems;
  const int u0 = gp.cta_u0[blockIdx.x], u1 = gp.cta_u0[blockIdx.x + 1];
  const int n_units = u1 - u0;
  const MbSmem lay = mb_smem_layout(S, MT, GRP, gp.res_stage_bytes);
  uint8_t* stages = smem;
  MbProblemArgs* tab = reinterpret_cast<MbProblemArgs*>(smem + lay.tab);
  float* rslot = reinterpret_cast<float*>(smem + lay.rslot);      // [2][256][8 MT] helpers' results
  uint8_t* rstage = smem + lay.rstage;                             // helpers' staging
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + lay.bars);   // [S] stage landed
  uint64_t* empty = full + S;                                      // [S] consumers released it
  uint64_t* res_full = empty + S;                                  // [2] helpers wrote the slot
  uint64_t* res_empty = res_full + 2;                              // [2] consumers read the slot
  uint64_t* staged = res_empty + 2;                                // helpers' bulk copies landed
  int* last_fill = reinterpret_cast<int*>(smem + lay.last_fill);   // [S] fills issued per stage

  // the problem table goes to shared memory in one step (every thread one word)
  {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(gp.prob);
    uint32_t* dst = reinterpret_cast<uint32_t*>(tab);
    const int words = NP * (int)(sizeof(MbProblemArgs) / 4);
    for (int i = threadIdx.x; i < words; i += kMbThreads) dst[i] = src[i];
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), kMbConsumerWarps);
      last_fill[i] = 0;
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&res_full[i]), kMbHelperWarps);
      mbar_init(smem_u32(&res_empty[i]), kMbConsumerWarps);
    }
    mbar_init(smem_u32(staged), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == kMbConsumerWarps && lane < NP)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.m[lane])) : "memory");
  if (GRP && warp == kMbConsumerWarps && lane >= 16 && lane - 16 < NP)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&ab_maps.m[lane - 16])) : "memory");
  __syncthreads();
  // the codes of the first stages are the library's and no kernel writes them: they may load before
  // the grid dependency wait; v and x in fragment order come from the prep kernel, after it
  if (warp == kMbConsumerWarps && lane == 0) {
    for (int i = 0; i < S && i < n_units; ++i) {
      const UnitPos up = unit_pos(tab, NP, (long long)u0 + i);
      const uint32_t bar = smem_u32(&full[i]);
      mbar_arrive_expect_tx(bar, (gp.fused && i == 0) ? kFill - (kMbChunkHead + MT * kMbXTileBytes) : kFill);
      tma_load_2d(smem_u32(stages + (size_t)i * kStage), &maps.m[up.p], up.ch * kChunkRowBytes, up.t * kMbTileRows,
                  bar);
      last_fill[i] = 1;
    }
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  if (gp.fused && warp < kMbConsumerWarps) {
    // the prep work, done by the consumer threads while the first code stages stream in: this CTA's
    // first unit's v and x straight into stage 0, then its share of every chunk's fragment-order v and
    // x and of x at the salient columns (global memory, for the later units of all CTAs), then an
    // arrival at the grid barrier that the producer and the helpers wait on before their bulk copies
    {
      const UnitPos up = unit_pos(tab, NP, u0);
      const MbPrepProblem pp = gp.prep.prob[up.p];
      if (SPLIT)
        prep_chunk_split(pp, gp.M, MT, up.ch, (int)threadIdx.x, rstage, stages + kMbCodeBytes, [] { consumers_sync(); });
      else
        prep_chunk(pp, gp.M, MT, up.ch, (int)threadIdx.x, rstage, stages + kMbCodeBytes, [] { consumers_sync(); });
      consumers_sync();
    }
    {
      for (int item = blockIdx.x; item < gp.prep.n_blocks; item += gridDim.x) {
        int pi = 0;
        while (pi + 1 < gp.prep.n_problems && item >= gp.prep.prob[pi + 1].block_begin) ++pi;
        const MbPrepProblem pp = gp.prep.prob[pi];
        const int local = item - pp.block_begin;
        if (local < pp.n_chunks && SPLIT)
          prep_chunk_split(pp, gp.M, MT, local, (int)threadIdx.x, rstage, pp.ws + (size_t)local * kMbChunkWsBytes,
                           [] { consumers_sync(); });
        else if (local < pp.n_chunks)
          prep_chunk(pp, gp.M, MT, local, (int)threadIdx.x, rstage, pp.ws + (size_t)local * kMbChunkWsBytes,
                     [] { consumers_sync(); });
        else
          prep_gather(pp, gp.M, local - pp.n_chunks, (int)threadIdx.x);
        consumers_sync();  // the scratch is free again
      }
    }
    if (threadIdx.x == 0) grid_arrive(gp.gbar);
  }

  if (warp > kMbConsumerWarps) {
    helper_role<MT, SPLIT>(tab, NP, u0, n_units, rslot, rstage, res_full, res_empty, staged, gp, warp - kMbConsumerWarps - 1,
                    lane, gp.status);
  } else if (warp == kMbConsumerWarps) {
    // ---------------------------------------------------------------- producer lane
    if (lane == 0) {
      // the chunks' fragment-order v and x were written by generic stores (the CTAs before the grid
      // barrier, or the prep kernel); the bulk copies read them through the async proxy
      asm volatile("fence.proxy.async.global;" ::: "memory");
      bool barrier_passed = !gp.fused;
      for (int i = 0; i < n_units; ++i) {
        const int st = i % S, ph = i / S;
        const UnitPos up = unit_pos(tab, NP, (long long)u0 + i);
        uint8_t* sb = stages + (size_t)st * kStage;
        const uint32_t bar = smem_u32(&full[st]);
        if (ph > 0) {
          if (!mbar_wait(smem_u32(&empty[st]), (uint32_t)((ph - 1) & 1), gp.status)) break;
          mbar_arrive_expect_tx(bar, kFill);
          tma_load_2d(smem_u32(sb), &maps.m[up.p], up.ch * kChunkRowBytes, up.t * kMbTileRows, bar);
          last_fill[st] = ph + 1;
        }
        if (!(gp.fused && i == 0)) {  // fused: unit 0's v and x were written by this CTA's consumers
          if (!barrier_passed) {
            grid_wait(gp.gbar, gp.gbar_target, gp.status);
            barrier_passed = true;
          }
          // stage 0 held generic stores of unit 0 before this copy overwrites it
          if (st == 0) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          bulk_load(smem_u32(sb + kMbCodeBytes), tab[up.p].ws + (size_t)up.ch * kMbChunkWsBytes,
                    (uint32_t)(kMbChunkHead + MT * kMbXTileBytes), bar);
        }
        if (GRP) {
          // the unit's alpha (and beta): 8 fp16 per row from column 8 ch (pairs) or 8 (ch / 2)
          const int xa = tab[up.p].bias ? 8 * up.ch : 8 * (up.ch >> 1);
          tma_load_2d(smem_u32(sb + kMbCodeBytes + kMbChunkHead + MT * kMbXTileBytes), &ab_maps.m[up.p], xa,
                      up.t * kMbTileRows, bar);
        }
      }
    }
  } else {
    // ---------------------------------------------------------------- consumers
    const int g = lane >> 2, q = lane & 3;
    const int tr = warp * 16 * kMbBlocks;  // first row of the warp's 16-row blocks
    const int tid = threadIdx.x;           // consumer index
    const int grid = gridDim.x;
    const int M = gp.M;
    float acc[2][kMbBlocks][MT][4], res[kMbBlocks][MT][4], run[kMbBlocks][MT][4];
#pragma unroll
    for (int e = 0; e < 2; ++e)
#pragma unroll
      for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
        for (int j = 0; j < MT; ++j)
#pragma unroll
          for (int k = 0; k < 4; ++k) acc[e][b][j][k] = res[b][j][k] = run[b][j][k] = 0.f;
    uint16_t al[kMbBlocks][2] = {};
    uint4 pw[kMbBlocks];   // MT = 1: the first partner's words of the split tile the range ends in
    bool pre = false;
    bool need_alpha = true;
    bool own_res = false;  // the helpers compute this tile's residual
    int kc = 0;            // helper result slots taken so far
    UnitPos c = unit_pos(tab, NP, u0);
    for (int i = 0; i < n_units; ++i) {
      const int u = u0 + i, st = i % S;
      const MbProblemArgs& a = tab[c.p];
      const int tile_row = c.t * kMbTileRows + tr;
      if (!GRP && need_alpha) {  // used at the tile's end; the loads complete during the decode
#pragma unroll
        for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int row = tile_row + 16 * b + 8 * h + g;
            al[b][h] = row < a.N ? __ldg(a.alpha + row) : (uint16_t)0;
          }
        need_alpha = false;
      }
      if (c.ch == 0) {
        // the tile's residual (Eq. 11) is added once, by the CTA that decodes its first chunk
        own_res = a.res_mode == kMbResHelpers;
        if (a.res_mode == kMbResPrep) {
          const float4* src = reinterpret_cast<const float4*>(a.yres + ((size_t)c.t * 256 + tid) * 4 * kMbBlocks * MT);
#pragma unroll
          for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
            for (int j = 0; j < MT; ++j) {
              const float4 r4 = __ldcg(src + b * MT + j);
              res[b][j][0] = r4.x;
              res[b][j][1] = r4.y;
              res[b][j][2] = r4.z;
              res[b][j][3] = r4.w;
            }
        }
      }
      if (MT == 1 && i == n_units - 1) {
        // the split tile this range ends in, when this CTA sums it: the first partner's partial rows,
        // loaded now so that they arrive during the decode
        const long long A = a.unit_begin + (long long)c.t * a.n_chunks, B = A + a.n_chunks;
        if (A >= u0 && B > u1) {
          const uint4* src = reinterpret_cast<const uint4*>(
              a.part + ((size_t)(blockIdx.x + 1) * 2 * kMbConsumerWarps * 32 + tid) * 4 * kMbBlocks * MT);
#pragma unroll
          for (int b = 0; b < kMbBlocks; ++b) pw[b] = part_load4(src + b);
          pre = true;
        }
      }
      const bool ok = mbar_wait(smem_u32(&full[st]), (uint32_t)((i / S) & 1), gp.status);
      if (!__all_sync(0xffffffffu, ok)) break;
      decode_unit<MT, GRP, SPLIT>(stages + (size_t)st * kStage, tr, g, q, lane, c.ch & 1, a.bias != 0, acc, run);
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[st]));

      // ---- tile epilogue once this CTA's part of tile c.t is done
      if (c.ch == a.n_chunks - 1 || u == u1 - 1) {
        const int t = c.t;
        if (own_res) {
          const int slot = kc & 1;
          const bool rok = mbar_wait(smem_u32(&res_full[slot]), (uint32_t)((kc >> 1) & 1), gp.status);
          if (!__all_sync(0xffffffffu, rok)) break;
          const float4* src = reinterpret_cast<const float4*>(rslot + ((size_t)slot * 256 + tid) * 8 * MT);
#pragma unroll
          for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
            for (int j = 0; j < MT; ++j) {
              const float4 r4 = src[b * MT + j];
              res[b][j][0] += r4.x;
              res[b][j][1] += r4.y;
              res[b][j][2] += r4.z;
              res[b][j][3] += r4.w;
            }
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&res_empty[slot]));
          ++kc;
          own_res = false;
        }
        // this CTA's part: alpha * acc / 2 + res (alpha scales only the ternary part), or with scale
        // groups the folded sum
        float part[kMbBlocks][MT][4];
#pragma unroll
        for (int b = 0; b < kMbBlocks; ++b) {
          const float fa0 = GRP ? 0.f : 0.5f * h2f(al[b][0]), fa1 = GRP ? 0.f : 0.5f * h2f(al[b][1]);
#pragma unroll
          for (int j = 0; j < MT; ++j) {
            if (GRP) {
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                part[b][j][e] = run[b][j][e] + res[b][j][e];
                run[b][j][e] = 0.f;
              }
            } else if (SPLIT) {  // the folded chunks, then alpha (entries 1 and 3 carry nothing)
              part[b][j][0] = fmaf(h2f(al[b][0]), run[b][j][0], res[b][j][0]);
              part[b][j][2] = fmaf(h2f(al[b][1]), run[b][j][2], res[b][j][2]);
              part[b][j][1] = part[b][j][3] = 0.f;
#pragma unroll
              for (int e = 0; e < 4; ++e) run[b][j][e] = 0.f;
            } else {
              part[b][j][0] = fa0 * (acc[0][b][j][0] + acc[1][b][j][0]) + res[b][j][0];
              part[b][j][1] = fa0 * (acc[0][b][j][1] + acc[1][b][j][1]) + res[b][j][1];
              part[b][j][2] = fa1 * (acc[0][b][j][2] + acc[1][b][j][2]) + res[b][j][2];
              part[b][j][3] = fa1 * (acc[0][b][j][3] + acc[1][b][j][3]) + res[b][j][3];
            }
          }
        }
        const long long A = a.unit_begin + (long long)t * a.n_chunks, B = A + a.n_chunks;
        bool write = true;
        if (!(A >= u0 && B <= u1)) {
          // split tile, summed in CTA order by the CTA that holds its first unit (bitwise
          // reproducible): every other contributor stores its partial rows in slot 0 of its
          // partial-row slots, each word XOR-ed with kPartEmpty (zero: not written), and carries on;
          // the first contributor reaches the tile at the end of its range, waits for each partner's
          // words (bounded), adds them and zeroes them, so every completed call leaves the slots zero
          const int bl = unit_owner(B - 1, gp.total_units, grid);
          if (A < u0) {
            uint4* mine = reinterpret_cast<uint4*>(
                a.part + ((size_t)blockIdx.x * 2 * kMbConsumerWarps * 32 + tid) * 4 * kMbBlocks * MT);
#pragma unroll
            for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
              for (int j = 0; j < MT; ++j)
                part_store4(mine + b * MT + j,
                            make_uint4(__float_as_uint(part[b][j][0]) ^ kPartEmpty, __float_as_uint(part[b][j][1]) ^ kPartEmpty,
                                       __float_as_uint(part[b][j][2]) ^ kPartEmpty, __float_as_uint(part[b][j][3]) ^ kPartEmpty));
            write = false;
          } else {
            bool timed_out = false;
            for (int cb = (int)blockIdx.x + 1; cb <= bl; ++cb) {
              uint4* src = reinterpret_cast<uint4*>(
                  a.part + ((size_t)cb * 2 * kMbConsumerWarps * 32 + tid) * 4 * kMbBlocks * MT);
              uint4 w[kMbBlocks][MT];
#pragma unroll
              for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
                for (int j = 0; j < MT; ++j)
                  w[b][j] = (MT == 1 && pre && cb == (int)blockIdx.x + 1) ? pw[b] : part_load4(src + b * MT + j);
#pragma unroll
              for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
                for (int j = 0; j < MT; ++j) {
                  if (!timed_out && !part_written4(w[b][j])) {
                    const unsigned long long t0 = global_ns();
                    do {
                      w[b][j] = part_load4(src + b * MT + j);
                      if (global_ns() - t0 > kWaitLimitNs) {
                        atomicExch(gp.status, (int)QTEA_ERR_TIMEOUT);
                        timed_out = true;
                        break;
                      }
                    } while (!part_written4(w[b][j]));
                  }
                  part[b][j][0] += __uint_as_float(w[b][j].x ^ kPartEmpty);
                  part[b][j][1] += __uint_as_float(w[b][j].y ^ kPartEmpty);
                  part[b][j][2] += __uint_as_float(w[b][j].z ^ kPartEmpty);
                  part[b][j][3] += __uint_as_float(w[b][j].w ^ kPartEmpty);
                  part_store4(src + b * MT + j, make_uint4(0u, 0u, 0u, 0u));  // empty again for the next call
                }
            }
          }
          pre = false;
        }
        if (write) {
#pragma unroll
          for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
            for (int j = 0; j < MT; ++j) {
              const int row0 = c.t * kMbTileRows + tr + 16 * b + g, row1 = row0 + 8;
              if (SPLIT) {  // batch row 4j + q in entries 0 (row g) and 2 (row g + 8)
                const int m = 4 * j + q;
                if (m < M && row0 < a.N) a.y[(size_t)m * a.N + row0] = part[b][j][0];
                if (m < M && row1 < a.N) a.y[(size_t)m * a.N + row1] = part[b][j][2];
                continue;
              }
              const int n0 = 8 * j + 2 * q;
              if (row0 < a.N) {
                if (n0 < M) a.y[(size_t)n0 * a.N + row0] = part[b][j][0];
                if (n0 + 1 < M) a.y[(size_t)(n0 + 1) * a.N + row0] = part[b][j][1];
              }
              if (row1 < a.N) {
                if (n0 < M) a.y[(size_t)n0 * a.N + row1] = part[b][j][2];
                if (n0 + 1 < M) a.y[(size_t)(n0 + 1) * a.N + row1] = part[b][j][3];
              }
            }
        }
#pragma unroll
        for (int e = 0; e < 2; ++e)
#pragma unroll
          for (int b = 0; b < kMbBlocks; ++b)
#pragma unroll
            for (int j = 0; j < MT; ++j)
#pragma unroll
              for (int k = 0; k < 4; ++k) acc[e][b][j][k] = res[b][j][k] = 0.f;
        need_alpha = true;
      }
      if (++c.ch == a.n_chunks) {
        c.ch = 0;
        if (++c.t == a.n_tiles) {
          c.t = 0;
          ++c.p;
        }
      }
    }
  }

  // no bulk copy may still be writing shared memory when the CTA exits (after a timeout the
  // consumers may not have waited for every fill)
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int s2 = 0; s2 < S; ++s2) {
      const int lf = last_fill[s2];
      if (lf > 0 && !mbar_wait(smem_u32(&full[s2]), (uint32_t)((lf - 1) & 1), gp.status)) break;
    }
  }
}

}  // namespace

size_t mb_smem_bytes(int S, int M, bool grp, int res_stage_bytes) {
  return mb_smem_layout(S, mb_mt(M), grp, res_stage_bytes).total;
}

// The six variants of the main kernel: (MT, GRP, SPLIT) in {(1, -, 1), (1, -, 0), (2, -, 0)}.
#define QTEA_MB_VARIANTS(X)                                                                                 \
  X(1, false, true) X(1, false, false) X(2, false, false) X(1, true, true) X(1, true, false) X(2, true, false)

cudaError_t mb_configure(size_t smem_optin, size_t* dyn_max) {
  cudaError_t e;
  size_t st = 0;
  cudaFuncAttributes a;
#define QTEA_MB_ATTR(MT, GRP, SPLIT)                                                                        \
  if ((e = cudaFuncGetAttributes(&a, qtea_gemv_mb_kernel<MT, GRP, SPLIT>)) != cudaSuccess) return e;      \
  st = a.sharedSizeBytes > st ? a.sharedSizeBytes : st;
  QTEA_MB_VARIANTS(QTEA_MB_ATTR)
#undef QTEA_MB_ATTR
  const size_t dyn = smem_optin > st ? smem_optin - st : 0;
  *dyn_max = dyn;
#define QTEA_MB_SET(MT, GRP, SPLIT)                                                                         \
  if ((e = cudaFuncSetAttribute(qtea_gemv_mb_kernel<MT, GRP, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                (int)dyn)) != cudaSuccess)                                                  \
    return e;
  QTEA_MB_VARIANTS(QTEA_MB_SET)
#undef QTEA_MB_SET
  return cudaSuccess;
}

size_t mb_prep_smem_bytes(int s, bool native) {
  const size_t E = native ? (size_t)s : (size_t)kMbResEntries;
  const size_t ris = native ? (size_t)((s + 3) / 4) : (size_t)kMbResEntries / 4;
  const size_t res = ((64 * E * 2 + 15) & ~(size_t)15) + ((64 * ris + 15) & ~(size_t)15) + 16 * ((E + 15) & ~(size_t)15) * 2;
  const size_t chunk = (size_t)kMbPrepScratch;
  return s > 0 && res > chunk ? res : chunk;
}

cudaError_t mb_prep_configure(size_t smem_optin) {
  cudaError_t e = cudaFuncSetAttribute(qtea_mb_prep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_optin);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(qtea_mb_prep_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
}

cudaError_t launch_mb_prep(const MbPrepGroup& g, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)g.n_blocks);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = g.smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, qtea_mb_prep_kernel, g);
}

cudaError_t launch_mb(const TensorMaps& maps, const TensorMaps& ab_maps, const MbGroupParams& p, bool grp, int grid,
                      size_t smem, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kMbThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeCooperative;  // fused: the CTAs wait on one another (grid barrier)
  attr[1].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.fused ? 2 : 1;
  const int mt = mb_mt(p.M);
  const bool split = p.split != 0;
  if (grp) {
    if (split) return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<1, true, true>, maps, ab_maps, p);
    if (mt == 1) return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<1, true, false>, maps, ab_maps, p);
    return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<2, true, false>, maps, ab_maps, p);
  }
  if (split) return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<1, false, true>, maps, ab_maps, p);
  if (mt == 1) return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<1, false, false>, maps, ab_maps, p);
  return cudaLaunchKernelEx(&cfg, qtea_gemv_mb_kernel<2, false, false>, maps, ab_maps, p);
}

}  // namespace qtea
