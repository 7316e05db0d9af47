// Device code shared by the batch-1 kernels (the stream-K kernel and the row-resident kernel):
// the fixed-point decode of 2-bit codes against byte planes of v*x, and the staging of a
// 512-column chunk's v*x as those planes. Included by CUDA sources only.
#pragma once

#include <cuda_fp16.h>

#include "qtea_internal.h"

namespace qtea {
namespace {

// Accumulators of one row for one chunk: [plane][column group]. A code word masked with
// 0x03030303 << 2k holds the codes of column group k in its byte lanes, scaled by 4^k (no shift).
template <int P>
struct RowAcc {
  int a[P][4];
};

// dp4a of unsigned code bytes with a signed plane (the top byte plane of X).
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
  int d;
  asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// One 32-bit word = 16 codes of one row. Plane registers of the word, in the order
// [group k][plane q] (group k = columns {k, 4+k, 8+k, 12+k} in byte lanes 0..3): for P = 3,
// P0 = {g0p0, g0p1, g0p2, g1p0}, P1 = {g1p1, g1p2, g2p0, g2p1}, P2 = {g2p2, g3p0, g3p1, g3p2};
// for P = 2, P0 = {g0p0, g0p1, g1p0, g1p1}, P1 = {g2p0, g2p1, g3p0, g3p1}. The top plane is
// signed, the others unsigned.
__device__ __forceinline__ void decode_word3(uint32_t w, const uint4& P0, const uint4& P1, const uint4& P2,
                                             RowAcc<3>& r) {
  const uint32_t g0 = w & 0x03030303u;  // columns 0,4,8,12 -> byte lanes, values c
  const uint32_t g1 = w & 0x0C0C0C0Cu;  // columns 1,5,9,13, values 4c
  const uint32_t g2 = w & 0x30303030u;  // columns 2,6,10,14, values 16c
  const uint32_t g3 = w & 0xC0C0C0C0u;  // columns 3,7,11,15, values 64c
  r.a[0][0] = (int)__dp4a(g0, P0.x, (unsigned)r.a[0][0]);
  r.a[1][0] = (int)__dp4a(g0, P0.y, (unsigned)r.a[1][0]);
  r.a[2][0] = dp4a_us(g0, P0.z, r.a[2][0]);
  r.a[0][1] = (int)__dp4a(g1, P0.w, (unsigned)r.a[0][1]);
  r.a[1][1] = (int)__dp4a(g1, P1.x, (unsigned)r.a[1][1]);
  r.a[2][1] = dp4a_us(g1, P1.y, r.a[2][1]);
  r.a[0][2] = (int)__dp4a(g2, P1.z, (unsigned)r.a[0][2]);
  r.a[1][2] = (int)__dp4a(g2, P1.w, (unsigned)r.a[1][2]);
  r.a[2][2] = dp4a_us(g2, P2.x, r.a[2][2]);
  r.a[0][3] = (int)__dp4a(g3, P2.y, (unsigned)r.a[0][3]);
  r.a[1][3] = (int)__dp4a(g3, P2.z, (unsigned)r.a[1][3]);
  r.a[2][3] = dp4a_us(g3, P2.w, r.a[2][3]);
}

__device__ __forceinline__ void decode_word2(uint32_t w, const uint4& P0, const uint4& P1, RowAcc<2>& r) {
  const uint32_t g0 = w & 0x03030303u;
  const uint32_t g1 = w & 0x0C0C0C0Cu;
  const uint32_t g2 = w & 0x30303030u;
  const uint32_t g3 = w & 0xC0C0C0C0u;
  r.a[0][0] = (int)__dp4a(g0, P0.x, (unsigned)r.a[0][0]);
  r.a[1][0] = dp4a_us(g0, P0.y, r.a[1][0]);
  r.a[0][1] = (int)__dp4a(g1, P0.z, (unsigned)r.a[0][1]);
  r.a[1][1] = dp4a_us(g1, P0.w, r.a[1][1]);
  r.a[0][2] = (int)__dp4a(g2, P1.x, (unsigned)r.a[0][2]);
  r.a[1][2] = dp4a_us(g2, P1.y, r.a[1][2]);
  r.a[0][3] = (int)__dp4a(g3, P1.z, (unsigned)r.a[0][3]);
  r.a[1][3] = dp4a_us(g3, P1.w, r.a[1][3]);
}

// sum_j c_j X_j of plane q: group k's accumulator is 4^k times its share, exactly divisible.
template <int P>
__device__ __forceinline__ int plane_sum(const RowAcc<P>& r, int q) {
  return r.a[q][0] + (r.a[q][1] >> 2) + (r.a[q][2] >> 4) + (r.a[q][3] >> 6);
}

// sum_j (c_j - 1) X_j over the chunk, exact: in int32 with two planes (|sum| < 2^25), in int64
// with three.
__device__ __forceinline__ float finish_chunk2(const RowAcc<2>& r, int sum_x) {
  return (float)(plane_sum<2>(r, 0) + (plane_sum<2>(r, 1) << 8) - sum_x);
}
__device__ __forceinline__ float finish_chunk3(const RowAcc<3>& r, long long sum_x) {
  return (float)((long long)plane_sum<3>(r, 0) + ((long long)plane_sum<3>(r, 1) << 8) +
                 ((long long)plane_sum<3>(r, 2) << 16) - sum_x);
}

// Decode one unit (two rows per lane, 32 words each) against the chunk's P byte planes.
// The next word's planes and the next 16 bytes of both rows are loaded while the current
// word decodes.
template <int P>
__device__ __forceinline__ void decode_unit(const uint4* row0, const uint4* row1, const uint4* pl, int sw,
                                            RowAcc<P>& a0, RowAcc<P>& a1) {
  constexpr int kW = (P == 3) ? 3 : 2;  // uint4 of planes per word (stride 3 in the slot)
#pragma unroll
  for (int k = 0; k < P; ++k)
#pragma unroll
    for (int g = 0; g < 4; ++g) a0.a[k][g] = a1.a[k][g] = 0;
  uint4 P0 = pl[0], P1 = pl[1], P2 = kW == 3 ? pl[2] : make_uint4(0, 0, 0, 0);
  uint4 c0 = row0[0 ^ sw], c1 = row1[0 ^ sw];
#pragma unroll 2  // two chunks per iteration: the code and plane registers alternate without copies
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

// x and v of columns 16*lane .. 16*lane+15 of one chunk, as fp16 pairs (zero beyond K).
struct ChunkLoads {
  uint32_t x[8], v[8];
};

__device__ __forceinline__ void load_chunk(const ProblemArgs& a, int ch, int lane, ChunkLoads& L) {
  const int col0 = ch * kChunkCols + lane * 16;
  if (a.vec_xv && col0 + 16 <= a.K) {
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

// Largest of the lanes' non-negative values: their bit patterns order as unsigned integers, so one
// warp reduction instruction serves.
__device__ __forceinline__ float warp_max(float v) {
  return __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(v)));
}

// Largest |xt[i]| of the lane's values whose bit in skip is clear, as a tree (a short chain).
__device__ __forceinline__ float lane_max(const float (&xt)[16], uint32_t skip) {
  float m[8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
    m[i] = fmaxf(((skip >> (2 * i)) & 1u) ? 0.f : fabsf(xt[2 * i]), ((skip >> (2 * i + 1)) & 1u) ? 0.f : fabsf(xt[2 * i + 1]));
#pragma unroll
  for (int w = 4; w; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) m[i] = fmaxf(m[i], m[i + w]);
  return m[0];
}

// 2^-(e+1) for amax in [2^e, 2^(e+1)) (2^126 for amax = 0): values up to amax scale into (-1, 1).
__device__ __forceinline__ float binade_scale(float amax) {
  return __uint_as_float((uint32_t)(253 - (int)((__float_as_uint(amax) >> 23) & 0xff)) << 23);
}

// Sum over the warp of the squares of the values whose bit in skip is clear, scaled by
// binade_scale(amax)^2 and then by 2^20, in integer units: a lane's share is below 16 * 2^20, so the
// warp's sum fits 32 bits and one warp reduction instruction serves. Truncation costs at most one
// unit per lane against a sum of at least 2^18 (the largest value alone): this feeds only the choice
// between 16- and 24-bit planes.
__device__ __forceinline__ unsigned warp_sq_units(const float (&xt)[16], uint32_t skip, float amax) {
  const float sc = binade_scale(amax);
  float q0 = 0.f, q1 = 0.f, q2 = 0.f, q3 = 0.f;  // four partial sums per lane (short chains)
#pragma unroll
  for (int i = 0; i < 16; i += 4) {
    const float z0 = xt[i] * sc, z1 = xt[i + 1] * sc, z2 = xt[i + 2] * sc, z3 = xt[i + 3] * sc;
    q0 = ((skip >> i) & 1u) ? q0 : fmaf(z0, z0, q0);
    q1 = ((skip >> (i + 1)) & 1u) ? q1 : fmaf(z1, z1, q1);
    q2 = ((skip >> (i + 2)) & 1u) ? q2 : fmaf(z2, z2, q2);
    q3 = ((skip >> (i + 3)) & 1u) ? q3 : fmaf(z3, z3, q3);
  }
  return __reduce_add_sync(0xffffffffu, __float2uint_rz(((q0 + q1) + (q2 + q3)) * 1048576.f));
}

// The fixed-point parameters of a staged chunk, the same on every lane of the staging warp.
struct ChunkStage {
  float scale;      // q
  int planes;       // 2 or 3
  int n_out;        // outliers taken out
  long long sum_x;  // sum of the fixed-point values
};

// The chunk's v*x as fixed point: byte planes of this lane's word, and the metadata.
//  * Outliers: in up to kOutlierRounds rounds, the elements above 1/16 of the largest |v*x| not yet
//    taken are taken, as long as at most kMaxOutliers are taken in all. A round of ordinary values
//    has hundreds above that threshold and ends the search, so only values at least 16 times above
//    the rest are ever taken. They get X = 0 in the planes and are listed in the metadata with
//    their exact v*x, which the consumers add per row in fp32.
//  * The remaining values set the quantum: their largest magnitude amax in [2^e, 2^(e+1)) gives
//    q = 2^(e-22) for 24 bits (|X| < 2^23) or q = 2^(e-14) for 16 bits (|X| < 2^15). 16 bits are
//    taken where the caller allows it and amax is within 8 times the root mean square of the
//    remaining values (no heavy tail that would coarsen the quantum of the others).
// kMeta: lane 0 also stores q, the plane count, the outlier count and the sum of X in the metadata
// (for consumers in other warps); the outlier list and the scale groups' sums are always stored.
// The returned values let a warp that decodes the chunk itself skip the shared-memory round trip.
template <bool kMeta = true>
__device__ __forceinline__ ChunkStage write_planes(const ProblemArgs& a, const ChunkLoads& L, uint8_t* ax,
                                                   int lane) {
  float xt[16];
#pragma unroll
  for (int i = 0; i < 8; ++i) {  // exact: fp16 x fp16 fits fp32
    xt[2 * i] = h2f((uint16_t)(L.v[i] & 0xffffu)) * h2f((uint16_t)(L.x[i] & 0xffffu));
    xt[2 * i + 1] = h2f((uint16_t)(L.v[i] >> 16)) * h2f((uint16_t)(L.x[i] >> 16));
  }
  float amax = warp_max(lane_max(xt, 0u));
  // the sum of squares for the usual case, no outliers, goes out beside the first round's count
  unsigned sq = warp_sq_units(xt, 0u, amax);
  uint32_t outm = 0;  // bit i: xt[i] is an outlier
  int n_out = 0;
#pragma unroll 1
  for (int round = 0; round < kOutlierRounds && amax > 0.f; ++round) {
    const float thr = amax * 0.0625f;
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) m |= (fabsf(xt[i]) > thr ? 1u : 0u) << i;
    m &= ~outm;
    const int c = (int)__reduce_add_sync(0xffffffffu, (unsigned)__popc(m));
    if (c > kMaxOutliers - n_out) break;
    outm |= m;
    n_out += c;
    amax = warp_max(lane_max(xt, outm));
  }
  if (n_out > 0) sq = warp_sq_units(xt, outm, amax);  // the remaining values, against their amax
  ChunkMeta* meta = reinterpret_cast<ChunkMeta*>(ax + kAuxMeta);
  if (n_out > 0) {  // list them: lane order, then element order
    const int mine = __popc(outm);
    int off = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, off, o);
      if (lane >= o) off += t;
    }
    off -= mine;
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if ((outm >> i) & 1u) {
        meta->out_col[off] = (uint16_t)(lane * 16 + i);
        meta->out_val[off] = xt[i];
        ++off;
      }
  }
  // amax^2 <= 64 * (sum of squares) / (values), both sides scaled by binade_scale(amax)^2:
  // 64 / 2^20 = 2^-14 turns the integer units back
  const float an = amax * binade_scale(amax);
  const bool two = a.act_bits == 16 && an * an * (float)(kChunkCols - n_out) <= (float)sq * 6.103515625e-05f;
  const int e = amax > 0.f ? (int)((__float_as_uint(amax) >> 23) & 0xff) - 127 : 0;
  const int qsh = two ? 14 : 22;
  const int xmax = two ? 32767 : 8388607;  // a value of amax rounds to at most 2^(qsh+1): clamp
  const float inv_q = __uint_as_float((uint32_t)(127 + qsh - e) << 23);
  int X[16];
  if (two) {
    // |v*x / q| <= 2^15 here: adding 1.5 * 2^23 rounds it to the nearest integer, ties to even, in
    // the low mantissa bits (exact for magnitudes below 2^22), the same value the conversion gives
    // (the product by the power of two inv_q is exact); an outlier's value is discarded
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float f = __fadd_rn(xt[i] * inv_q, 12582912.0f);
      X[i] = ((outm >> i) & 1u) ? 0 : min(__float_as_int(f) - 0x4B400000, xmax);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 16; ++i) X[i] = ((outm >> i) & 1u) ? 0 : min(__float2int_rn(xt[i] * inv_q), xmax);
  }
  // |sx| < 16 * 2^23 per lane
  const int sx = (((X[0] + X[1]) + (X[2] + X[3])) + ((X[4] + X[5]) + (X[6] + X[7]))) +
                 (((X[8] + X[9]) + (X[10] + X[11])) + ((X[12] + X[13]) + (X[14] + X[15])));
  // plane register (k, q): byte q of X[k], X[4 + k], X[8 + k], X[12 + k] in byte lanes 0 .. 3
  auto plane_reg = [&](int k, int q) {
    const uint32_t sel = (uint32_t)q | ((uint32_t)(4 + q) << 4);
    const uint32_t lo = __byte_perm((uint32_t)X[k], (uint32_t)X[4 + k], sel);
    const uint32_t hi = __byte_perm((uint32_t)X[8 + k], (uint32_t)X[12 + k], sel);
    return __byte_perm(lo, hi, 0x5410);
  };
  uint4* dst = reinterpret_cast<uint4*>(ax + (size_t)lane * kPlaneBytesPerWord);
  if (two) {
    dst[0] = make_uint4(plane_reg(0, 0), plane_reg(0, 1), plane_reg(1, 0), plane_reg(1, 1));
    dst[1] = make_uint4(plane_reg(2, 0), plane_reg(2, 1), plane_reg(3, 0), plane_reg(3, 1));
  } else {
    dst[0] = make_uint4(plane_reg(0, 0), plane_reg(0, 1), plane_reg(0, 2), plane_reg(1, 0));
    dst[1] = make_uint4(plane_reg(1, 1), plane_reg(1, 2), plane_reg(2, 0), plane_reg(2, 1));
    dst[2] = make_uint4(plane_reg(2, 2), plane_reg(3, 0), plane_reg(3, 1), plane_reg(3, 2));
  }
  if (a.gflags & kScaleGroups) {  // per 128-column group (lanes 8k .. 8k+7): sum of X, and sum of x for beta
    int gs = sx;
    float xs = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i)
      xs += h2f((uint16_t)(L.x[i] & 0xffffu)) + h2f((uint16_t)(L.x[i] >> 16));
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
      gs += __shfl_xor_sync(0xffffffffu, gs, o);
      xs += __shfl_xor_sync(0xffffffffu, xs, o);
    }
    if ((lane & 7) == 0) {
      meta->gsum_x[lane >> 3] = gs;
      meta->gsx[lane >> 3] = xs;
    }
  }
  // the chunk's sum of X, exact: the lanes' sums split into 16-bit halves, each summed by one warp
  // reduction instruction (|sum| < 2^32 in 24-bit mode)
  const unsigned s_lo = __reduce_add_sync(0xffffffffu, (unsigned)sx & 0xFFFFu);
  const int s_hi = (int)__reduce_add_sync(0xffffffffu, (unsigned)(sx >> 16));
  ChunkStage cs;
  cs.scale = __uint_as_float((uint32_t)(127 + e - qsh) << 23);  // q
  cs.planes = two ? 2 : 3;
  cs.n_out = n_out;
  cs.sum_x = (long long)s_hi * 65536 + (long long)s_lo;
  if (kMeta && lane == 0) {
    meta->scale = cs.scale;
    meta->planes = cs.planes;
    meta->sum_x = cs.sum_x;
    meta->n_out = cs.n_out;
  }
  return cs;
}

// x at the salient columns of entries e0 .. e0+31 (lane j holds entry e0 + j, zero past e_end).
__device__ __forceinline__ float gather_salient_x(const ProblemArgs& a, int e0, int e_end, int lane) {
  const int e = e0 + lane;
  if (e >= e_end) return 0.f;
  int col = __ldg(a.sal + e);
  col = col < 0 ? 0 : (col >= a.K ? a.K - 1 : col);
  return h2f(__ldg(a.x + col));
}

}  // namespace
}  // namespace qtea
