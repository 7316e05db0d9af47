// Batch-1 QTEA GEMV for sm_103a: y = alpha * (T . (v*x)) + sparse 1:4 residual, for one or
// several independent problems in one launch.
//
// Computes Eq. 10 (one alpha per row, beta = 0) plus Eq. 11 of the QTEA paper (Sec. 3.5).
// Design:
//  * Grouped persistent stream-K: the (problem, 512-row tile, 512-column chunk) units of all
//    problems form one sequence; one CTA per SM takes an equal contiguous share, so every SM
//    streams the same number of weight bytes and one launch amortises its fixed costs over
//    all problems.
//  * Roles: eight consumer warps decode from shared memory only, each lane owning two rows of
//    the tile (no cross-lane reduction). One producer lane keeps S code stages filled by TMA
//    (two 256 x 128-byte boxes per unit, 128-byte swizzle). Three helper warps take the units
//    round-robin and write each unit's auxiliary slot, in a ring of six: the chunk's v*x in
//    fixed point and the unit's share of the residual as one sum per row. A helper starts a unit
//    as soon as its slot is free, five units ahead of the consumers, so its loads are hidden.
//  * Decode: v*x (the column rescale of Sec. 3.3, fused into staging as the paper fuses it
//    into its LUT precompute) is held per 512-column chunk as 24-bit fixed point split into
//    three byte planes (or 16-bit, two planes, where the caller allows it and the chunk has no
//    dominant outlier). Codes are masked four at a time into byte lanes and multiplied with
//    dp4a, so sum_j c_j X_j is exact in integers; the ternary value is c - 1, whose
//    contribution is removed with the chunk's sum of X.
//  * Residual (Eq. 11): a tile's salient entries are split over its chunks by index, in blocks
//    of 8 (chunk ch of nc takes blocks [ch*nb/nc, (ch+1)*nb/nc)), so no search of the salient
//    list is needed and the work follows the weight stream. The values are never scaled by
//    alpha or v.
//  * Split tiles are summed in CTA order, so results are bitwise reproducible, by the CTA holding
//    the tile's first unit: the others store their partial rows (self-validating words: zero means
//    not written) and carry on without waiting; the first reaches the tile at the end of its range,
//    loads its first partner's rows before its last decode, and zeroes what it read.
//  * Programmatic dependent launch: before griddepcontrol.wait a CTA only initialises its
//    barriers, starts the TMA of its first units' codes when the library owns them (a layout's
//    packed codes, which no kernel writes after packing; caller-owned codes are fetched after the
//    wait), and prefetches into L2 the lines of x and v those units read (a prefetch reads no
//    value). Everything else the caller owns (x, v, alpha, the residual, y) and the split-tile
//    workspace is touched after the wait. Each CTA lets the next launch start once it is running.
// Every wait on an mbarrier is bounded: after ~2 s the waiting thread records
// QTEA_ERR_TIMEOUT in the status word and its role stops.
#include <cuda_fp16.h>

#include "qtea_internal.h"
#include "qtea_m1_device.h"

namespace qtea {
namespace {

// CTA whose range contains unit u.
__device__ __forceinline__ int unit_owner(long long u, long long total, int grid) {
  return (int)(((u + 1) * grid - 1) / total);
}

struct UnitPos {
  int p, t, ch;  // problem, tile, chunk
};

__device__ __forceinline__ UnitPos unit_pos(const ProblemArgs* tab, int n_problems, long long u) {
  int p = 0;
  while (p + 1 < n_problems && u >= tab[p + 1].unit_begin) ++p;
  const int v = (int)(u - tab[p].unit_begin);
  const int nc = tab[p].n_chunks;
  const int t = v / nc;
  return {p, t, v - t * nc};
}

// The two TMA boxes of unit (t, ch) into ring stage `dst`, completing on `bar`.
// The codes are read once per call: their lines are the first L2 evicts.
__device__ __forceinline__ void issue_unit(const CUtensorMap* map, int t, int ch, uint32_t dst, uint32_t bar) {
  const uint64_t pol = l2_evict_first_policy();
  mbar_arrive_expect_tx(bar, kStageBytes);
  tma_load_2d_hint(dst, map, ch * kChunkRowBytes, t * kTileRows, bar, pol);
  tma_load_2d_hint(dst + kBoxBytes, map, ch * kChunkRowBytes, t * kTileRows + kBoxRows, bar, pol);
}

// ---------------------------------------------------------------- decode (consumers)

// Scale groups of 128 columns: the unit's decode finished per group (every 8 words), each group's
// exact sum of T X scaled by q and its row's alpha, plus beta times the group's sum of x.
template <int P>
__device__ __forceinline__ void decode_unit_grouped(const uint4* row0, const uint4* row1, const uint4* pl, int sw,
                                                    const ChunkMeta* mp, float scale, const uint32_t (&g0)[4],
                                                    const uint32_t (&g1)[4], float& f0, float& f1) {
  constexpr int kW = (P == 3) ? 3 : 2;
  uint4 P0 = pl[0], P1 = pl[1], P2 = kW == 3 ? pl[2] : make_uint4(0, 0, 0, 0);
  uint4 c0 = row0[0 ^ sw], c1 = row1[0 ^ sw];
  float e0[4], e1[4];  // exact group sums of T X of both rows
#pragma unroll 1
  for (int g = 0; g < 4; ++g) {
    RowAcc<P> a0, a1;
#pragma unroll
    for (int k = 0; k < P; ++k)
#pragma unroll
      for (int q = 0; q < 4; ++q) a0.a[k][q] = a1.a[k][q] = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int jj = 2 * g + h;
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
    const int gsx = mp->gsum_x[g];
    float d0, d1;
    if constexpr (P == 2) {
      d0 = finish_chunk2(a0, gsx);
      d1 = finish_chunk2(a1, gsx);
    } else {
      d0 = finish_chunk3(a0, (long long)gsx);
      d1 = finish_chunk3(a1, (long long)gsx);
    }
    // kept per group (registers selected by index, not an indexed array)
    if (g == 0) { e0[0] = d0; e1[0] = d1; }
    else if (g == 1) { e0[1] = d0; e1[1] = d1; }
    else if (g == 2) { e0[2] = d0; e1[2] = d1; }
    else { e0[3] = d0; e1[3] = d1; }
  }
  // alpha (low half) and beta (high half) of each group, used only now: their loads, issued before
  // the decode, have had the whole unit to arrive
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const float sx = mp->gsx[g];
    f0 = fmaf(h2f((uint16_t)(g0[g] & 0xffffu)) * scale, e0[g], fmaf(h2f((uint16_t)(g0[g] >> 16)), sx, f0));
    f1 = fmaf(h2f((uint16_t)(g1[g] & 0xffffu)) * scale, e1[g], fmaf(h2f((uint16_t)(g1[g] >> 16)), sx, f1));
  }
}

// ---------------------------------------------------------------- staging (helpers)

// Scalar loads of a residual block, for shapes or pointers the vector loads cannot serve.
struct ResBlock {
  uint4 rv;     // 8 fp16 values
  uint32_t rp;  // 8 positions, 2 bits each
};

__device__ __noinline__ ResBlock load_block_scalar(const uint16_t* rvals, const uint8_t* ridx, int s, int q, int e0) {
  const int rs = (s + 3) >> 2;
  uint32_t h[8];
  uint32_t pos = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int e = e0 + j;
    h[j] = e < s ? __ldg(rvals + (size_t)q * s + e) : 0u;
    const uint32_t pb = e < s ? __ldg(ridx + (size_t)q * rs + e / 4) : 0u;
    pos |= ((pb >> (2 * (e & 3))) & 3u) << (2 * j);
  }
  ResBlock b;
  b.rv = make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16), h[6] | (h[7] << 16));
  b.rp = pos;
  return b;
}

// Values and positions of residual block b (entries 8b .. 8b+7) of group q.
__device__ __forceinline__ void load_block(const ProblemArgs& a, int q, int b, uint4& rv, uint32_t& rp) {
  rv = make_uint4(0, 0, 0, 0);
  rp = 0;
  if (q >= (a.N >> 2)) return;
  const int e0 = b * kResBlock;
  if (a.vec_res) {
    rv = __ldg(reinterpret_cast<const uint4*>(a.rvals + (size_t)q * a.s + e0));
    rp = __ldg(reinterpret_cast<const uint16_t*>(a.ridx + (size_t)q * ((a.s + 3) >> 2) + e0 / 4));
  } else {
    const ResBlock blk = load_block_scalar(a.rvals, a.ridx, a.s, q, e0);
    rv = blk.rv;
    rp = blk.rp;
  }
}

// Stage unit (t, ch) of problem *pa into auxiliary slot ax. First the planes and metadata, which
// need x and v only, then (after the arrival on planes_bar) the residual sums of the tile's 512
// rows over the unit's salient blocks: the consumers add those one unit later. The residual loads
// go out after the planes are published: issued earlier, they queue in front of the x and v loads
// behind the code stream and delay the planes. Lane owns residual groups lane + 32k.
__device__ __noinline__ void stage_unit(const ProblemArgs* pa, int t, int ch, uint8_t* ax, int lane,
                                        uint32_t planes_bar, float4* onehot) {
  const ProblemArgs a = *pa;
  {
    ChunkLoads L;
    load_chunk(a, ch, lane, L);
    write_planes(a, L, ax, lane);
  }
  mbar_arrive(planes_bar);

  const int nb = (a.s + kResBlock - 1) / kResBlock;
  const int b0 = (int)((long long)ch * nb / a.n_chunks), b1 = (int)((long long)(ch + 1) * nb / a.n_chunks);
  const int e_end = min(b1 * kResBlock, a.s);
  const int qb = t * (kTileRows / 4) + lane;
  // the salient indices and the first two residual blocks go out together; x at the salient
  // columns follows as soon as the indices arrive
  const bool has_entry = b0 * kResBlock + lane < e_end;  // lane j: entry 8 * b0 + j of the first window
  int col = has_entry ? __ldg(a.sal + b0 * kResBlock + lane) : 0;
  uint4 rvA[4], rvB[4];
  uint32_t rpA[4], rpB[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    rvA[k] = rvB[k] = make_uint4(0, 0, 0, 0);
    rpA[k] = rpB[k] = 0;
    if (b0 < b1) load_block(a, qb + 32 * k, b0, rvA[k], rpA[k]);
    if (b0 + 1 < b1) load_block(a, qb + 32 * k, b0 + 1, rvB[k], rpB[k]);
  }
  col = col < 0 ? 0 : (col >= a.K ? a.K - 1 : col);
  float xs = has_entry ? h2f(__ldg(a.x + col)) : 0.f;

  float acc[4][4];
#pragma unroll
  for (int k = 0; k < 4; ++k) acc[k][0] = acc[k][1] = acc[k][2] = acc[k][3] = 0.f;
#pragma unroll 1
  for (int b = b0; b < b1; ++b) {
    const int w = (b - b0) & 3;  // block within the 32-entry window of xs
    {
      // lane 4j + p writes T[j][p] = x_j * e_p for the block's entries j
      const float xj = __shfl_sync(0xffffffffu, xs, w * kResBlock + (lane >> 2));
      const int pp = lane & 3;
      onehot[lane] = make_float4(pp == 0 ? xj : 0.f, pp == 1 ? xj : 0.f, pp == 2 ? xj : 0.f, pp == 3 ? xj : 0.f);
      __syncwarp();
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t wd = (j < 2) ? rvA[k].x : (j < 4) ? rvA[k].y : (j < 6) ? rvA[k].z : rvA[k].w;
        const float rr = h2f((uint16_t)((j & 1) ? (wd >> 16) : (wd & 0xffffu)));
        const float4 oh = onehot[4 * j + (int)((rpA[k] >> (2 * j)) & 3u)];
        acc[k][0] = fmaf(rr, oh.x, acc[k][0]);
        acc[k][1] = fmaf(rr, oh.y, acc[k][1]);
        acc[k][2] = fmaf(rr, oh.z, acc[k][2]);
        acc[k][3] = fmaf(rr, oh.w, acc[k][3]);
      }
    }
    __syncwarp();  // every lane has read the table before the next block rewrites it
    // next block: B moves to A, the one after it is loaded into B; a new window of x every 4
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      rvA[k] = rvB[k];
      rpA[k] = rpB[k];
      if (b + 2 < b1) load_block(a, qb + 32 * k, b + 2, rvB[k], rpB[k]);
    }
    if (w == 3 && b + 1 < b1) xs = gather_salient_x(a, (b + 1) * kResBlock, e_end, lane);
  }
  float4* res = reinterpret_cast<float4*>(ax + kAuxRes);
#pragma unroll
  for (int k = 0; k < 4; ++k) res[lane + 32 * k] = make_float4(acc[k][0], acc[k][1], acc[k][2], acc[k][3]);
}

// ---------------------------------------------------------------- roles

struct Ring {
  uint8_t* codes;         // [S][kStageBytes]
  uint8_t* aux;           // [kAuxSlots][kAuxBytes]
  float4* onehot;         // [kHelperWarps][kResBlock * 4]
  const ProblemArgs* tab; // [n_problems], copied from the kernel parameters
  uint64_t* full_c;       // [S] codes landed
  uint64_t* empty_c;      // [S] consumers released the code stage
  uint64_t* planes_a;     // [kAuxSlots] planes and metadata of the auxiliary slot written
  uint64_t* full_a;       // [kAuxSlots] residual sums of the auxiliary slot written
  uint64_t* empty_a;      // [kAuxSlots] consumers released the auxiliary slot
  int* last_fill;         // [S] number of fills issued into each code stage
  int S, n_problems;
};

// The first fill of every code stage.
__device__ __forceinline__ void first_fills(const TensorMaps& maps, const Ring& r, int u0, int n_units) {
  for (int i = 0; i < r.S && i < n_units; ++i) {
    const UnitPos up = unit_pos(r.tab, r.n_problems, (long long)u0 + i);
    issue_unit(&maps.m[up.p], up.t, up.ch, smem_u32(r.codes + (size_t)i * kStageBytes), smem_u32(&r.full_c[i]));
    r.last_fill[i] = 1;
  }
}

// The producer lane: keeps the code stages filled. Fills 0 .. S-1 were issued before the grid
// dependency wait.
__device__ __noinline__ void producer_role(const TensorMaps& maps, const Ring r, int u0, int n_units, int* status) {
  for (int i = r.S; i < n_units; ++i) {
    const int st = i % r.S, fill = i / r.S;
    if (!mbar_wait(smem_u32(&r.empty_c[st]), (uint32_t)((fill - 1) & 1), status)) break;
    const UnitPos up = unit_pos(r.tab, r.n_problems, (long long)u0 + i);
    issue_unit(&maps.m[up.p], up.t, up.ch, smem_u32(r.codes + (size_t)st * kStageBytes), smem_u32(&r.full_c[st]));
    r.last_fill[st] = fill + 1;
  }
}

// Helper warp h: units h, h + 3, ...; unit i uses auxiliary slot i % 6, so slot h and slot h + 3
// belong to helper h alone and its waits on them come in order (a parity wait could not tell a
// phase two ahead from the current one).
__device__ __noinline__ void helper_role(const Ring r, int u0, int n_units, int h, int lane, int* status) {
  for (int i = h; i < n_units; i += kHelperWarps) {
    const int slot = i % kAuxSlots, fill = i / kAuxSlots;
    if (fill > 0) {
      const bool ok = mbar_wait(smem_u32(&r.empty_a[slot]), (uint32_t)((fill - 1) & 1), status);
      if (!__all_sync(0xffffffffu, ok)) break;
    }
    const UnitPos up = unit_pos(r.tab, r.n_problems, (long long)u0 + i);
    stage_unit(&r.tab[up.p], up.t, up.ch, r.aux + (size_t)slot * kAuxBytes, lane, smem_u32(&r.planes_a[slot]),
               r.onehot + h * (kOneHotBytes / 16));
    mbar_arrive(smem_u32(&r.full_a[slot]));
  }
}

// Residual sums of the auxiliary slot: wait until the helper has written them, return the lane's
// two rows, release the slot.
__device__ __forceinline__ bool take_residual(const Ring& r, int slot, uint32_t parity, int ra, int lane,
                                              float& res0, float& res1, int* status) {
  const bool ok = mbar_wait(smem_u32(&r.full_a[slot]), parity, status);
  if (!__all_sync(0xffffffffu, ok)) return false;
  const float* res = reinterpret_cast<const float*>(r.aux + (size_t)slot * kAuxBytes + kAuxRes);
  res0 = res[ra];
  res1 = res[ra + 32];
  __syncwarp();
  if (lane == 0) mbar_arrive(smem_u32(&r.empty_a[slot]));
  return true;
}

// A tile whose last unit this CTA has decoded: its lane rows' ternary sums, residual sums so far and
// alpha bits, held until the residual of that last unit is in.
struct DoneTile {
  float y0, y1, r0, r1;
  uint16_t al0, al1;
  int p, t;
};

// Partial sums of split tiles are stored XOR-ed with this NaN bit pattern, so that zeroed memory
// reads as "not written yet" and every 4-byte word validates itself (no result has this pattern):
// a reader needs no flag and no fence, only strong loads of the words (each is single-copy atomic).
constexpr uint32_t kPartEmpty = 0x7FBADBADu;

// Loads and stores of those words are strong (relaxed, GPU scope): a weak load may keep returning a
// stale copy of the line (the two dies' L2 partitions), so it need not ever see another CTA's store.
__device__ __forceinline__ void part_store_bits(float* p, unsigned w) {
  asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(w) : "memory");
}
__device__ __forceinline__ void part_store(float* p, float v) { part_store_bits(p, __float_as_uint(v) ^ kPartEmpty); }
__device__ __forceinline__ unsigned part_load(const float* p) {
  unsigned w;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(w) : "l"(p) : "memory");
  return w;
}

// The split tile that this CTA's range ends in, when this CTA holds its first unit (and so sums
// it): the first partner's words of the lane's rows, loaded before the CTA's last decode so that,
// when that partner holds the tile's last units (stored at the start of its range), they have
// arrived when the sum is formed.
struct EndTile {
  bool pre = false;
  unsigned w0 = 0u, w1 = 0u;        // partner blockIdx.x + 1's stored words of rows ra, ra + 32
};

// Write the tile's rows: directly when this CTA holds all of the tile's units, else through the
// split-tile workspace, summed in CTA order (bitwise reproducible) by the CTA that holds the tile's
// first unit. Every other contributor stores its partial rows in slot 0 of its workspace rows,
// encoded (part_store), and carries on without waiting, so its SM is free for the next launch
// sooner. The first contributor decodes the tile's first chunks at the end of its range; it then
// waits for each partner's words (bounded), adds them, and zeroes them: every completed call leaves
// the workspace zero, the start state. (Measured against a last-arriver atomic counter, Llama3-8B
// layer step: 17.5 against 18.7 us; gate_proj alone 9.0 against 10.1 us; down_proj alone, 19 CTAs
// per tile, 11.1 against 10.2 us.)
__device__ __forceinline__ void tile_epilogue(const ProblemArgs& a, const DoneTile& d, long long total, int u0,
                                              int u1, int ra, const EndTile& et, int* status) {
  const int N = a.N, t = d.t;
  const int row0g = t * kTileRows + ra, row1g = row0g + 32;
  const float val0 = h2f(d.al0) * d.y0 + d.r0;
  const float val1 = h2f(d.al1) * d.y1 + d.r1;
  const long long A = a.unit_begin + (long long)t * a.n_chunks, B = A + a.n_chunks;
  float* y = a.y;
  if (A >= u0 && B <= u1) {
    if (row0g < N) y[row0g] = val0;
    if (row1g < N) y[row1g] = val1;
    return;
  }
  const int grid = gridDim.x;
  float* ws = a.ws;
  const int bl = unit_owner(B - 1, total, grid);
  if (A < u0) {
    part_store(ws + (size_t)blockIdx.x * 2 * kTileRows + ra, val0);
    part_store(ws + (size_t)blockIdx.x * 2 * kTileRows + ra + 32, val1);
    return;
  }
  // the partners' words in batches of eight, all loads of a batch in flight together, then each
  // partner in CTA order: waited for (bounded) if not yet written, added, zeroed for the next call
  float s0 = val0, s1 = val1;
  bool timed_out = false;
  for (int cb0 = (int)blockIdx.x + 1; cb0 <= bl; cb0 += 8) {
    unsigned w[8][2];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int cb = cb0 + k;
      w[k][0] = w[k][1] = 0u;
      if (cb > bl) continue;
      const float* src = ws + (size_t)cb * 2 * kTileRows;
      if (cb == (int)blockIdx.x + 1 && et.pre) {  // loaded before the last decode
        w[k][0] = et.w0;
        w[k][1] = et.w1;
      }
      if (w[k][0] == 0u) w[k][0] = part_load(src + ra);
      if (w[k][1] == 0u) w[k][1] = part_load(src + ra + 32);
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int cb = cb0 + k;
      if (cb > bl) break;
      float* src = ws + (size_t)cb * 2 * kTileRows;
      unsigned w0 = w[k][0], w1 = w[k][1];
      if ((w0 == 0u || w1 == 0u) && !timed_out) {
        const unsigned long long t0 = global_ns();
        while (w0 == 0u || w1 == 0u) {
          if (w0 == 0u) w0 = part_load(src + ra);
          if (w1 == 0u) w1 = part_load(src + ra + 32);
          if (global_ns() - t0 > kWaitLimitNs) {
            atomicExch(status, (int)QTEA_ERR_TIMEOUT);
            timed_out = true;
            break;
          }
        }
      }
      s0 += __uint_as_float(w0 ^ kPartEmpty);
      s1 += __uint_as_float(w1 ^ kPartEmpty);
      part_store_bits(src + ra, 0u);  // empty again for the next call
      part_store_bits(src + ra + 32, 0u);
    }
  }
  if (row0g < N) y[row0g] = s0;
  if (row1g < N) y[row1g] = s1;
}

// The consumers take the units in order. A unit's residual sums, and for the last unit of a tile
// the tile's epilogue, wait until the next unit has been decoded, so the helpers' residual work is
// not waited for right after each decode; the sums are still added in unit order, so results stay
// bitwise reproducible.
template <int GM>
__device__ __forceinline__ void consumer_role(const Ring r, long long total, int u0, int u1,
                                           int warp, int lane, int* status) {
  const int n_units = u1 - u0;
  const int ra = warp * 64 + lane;  // tile rows owned by this lane: ra and ra + 32
  const int sw = lane & 7;          // 128-byte swizzle phase of both rows
  float yacc0 = 0.f, yacc1 = 0.f, racc0 = 0.f, racc1 = 0.f;
  uint16_t al0 = 0, al1 = 0;  // raw fp16 bits: converted at the tile's end, so no wait on the load here
  bool need_alpha = true;
  UnitPos c = unit_pos(r.tab, r.n_problems, u0);
  int st = 0, slot = 0;             // code stage and auxiliary slot of unit i
  uint32_t ph_c = 0, ph_a = 0;      // parity of their current fill
  int pend = -1;                    // auxiliary slot of the previous unit (residual not yet added)
  uint32_t pend_ph = 0;
  bool done = false;                // the previous unit ended a tile: its epilogue is pending
  DoneTile dt;
  EndTile et;

  for (int i = 0; i < n_units; ++i) {
    const int u = u0 + i;
    const ProblemArgs& a = r.tab[c.p];
    const int n_chunks = a.n_chunks, N = a.N;
    // GM: 0 no problem of the launch has scale groups, 2 every one has, 1 some have
    const bool grouped = GM == 2 || (GM == 1 && (a.gflags & kScaleGroups) != 0);
    const bool gbias = (a.gflags & kScaleBias) != 0, gvec = (a.gflags & kScaleVec) != 0;
    if (need_alpha) {  // used at the tile's end: unconditional loads (rows clamped), so nothing waits here
      if (grouped) {   // alpha is applied per group in the decode
        al0 = al1 = (uint16_t)0x3C00u;  // 1.0
      } else {
        al0 = __ldg(a.alpha + min(c.t * kTileRows + ra, N - 1));
        al1 = __ldg(a.alpha + min(c.t * kTileRows + ra + 32, N - 1));
      }
      need_alpha = false;
    }
    uint32_t gab0[4], gab1[4];  // scale groups: (alpha, beta) bits of the unit's four groups, both rows
    if (grouped) {
      const int r0 = min(c.t * kTileRows + ra, N - 1), r1 = min(c.t * kTileRows + ra + 32, N - 1);
      const int st_ = gbias ? 2 : 1;
      if (gvec && gbias) {  // (alpha, beta) of the four groups: one 16-byte load per row
        const uint4 v0 = __ldg(reinterpret_cast<const uint4*>(a.alpha + ((size_t)r0 * a.G + 4 * c.ch) * 2));
        const uint4 v1 = __ldg(reinterpret_cast<const uint4*>(a.alpha + ((size_t)r1 * a.G + 4 * c.ch) * 2));
        gab0[0] = v0.x; gab0[1] = v0.y; gab0[2] = v0.z; gab0[3] = v0.w;
        gab1[0] = v1.x; gab1[1] = v1.y; gab1[2] = v1.z; gab1[3] = v1.w;
      } else if (gvec) {         // alpha of the four groups: one 8-byte load per row
        const uint2 v0 = __ldg(reinterpret_cast<const uint2*>(a.alpha + (size_t)r0 * a.G + 4 * c.ch));
        const uint2 v1 = __ldg(reinterpret_cast<const uint2*>(a.alpha + (size_t)r1 * a.G + 4 * c.ch));
        gab0[0] = v0.x & 0xffffu; gab0[1] = v0.x >> 16; gab0[2] = v0.y & 0xffffu; gab0[3] = v0.y >> 16;
        gab1[0] = v1.x & 0xffffu; gab1[1] = v1.x >> 16; gab1[2] = v1.y & 0xffffu; gab1[3] = v1.y >> 16;
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int g = min((4 * c.ch + k) / a.gdiv, a.G - 1);
          const uint16_t* s0 = a.alpha + ((size_t)r0 * a.G + g) * st_;
          const uint16_t* s1 = a.alpha + ((size_t)r1 * a.G + g) * st_;
          gab0[k] = (uint32_t)__ldg(s0) | (gbias ? (uint32_t)__ldg(s0 + 1) << 16 : 0u);
          gab1[k] = (uint32_t)__ldg(s1) | (gbias ? (uint32_t)__ldg(s1 + 1) << 16 : 0u);
        }
      }
    }
    if (i == n_units - 1) {
      // the split tile this range ends in, when this CTA sums it: the first partner's words, loaded
      // now so that they arrive during the decode
      const long long A = a.unit_begin + (long long)c.t * n_chunks, B = A + n_chunks;
      if (A >= u0 && B > u1) {
        const float* src = a.ws + (size_t)(blockIdx.x + 1) * 2 * kTileRows;
        et.pre = true;
        et.w0 = part_load(src + ra);
        et.w1 = part_load(src + ra + 32);
      }
    }
    bool ok = mbar_wait(smem_u32(&r.full_c[st]), ph_c, status);
    ok = ok && mbar_wait(smem_u32(&r.planes_a[slot]), ph_a, status);
    if (!__all_sync(0xffffffffu, ok)) return;

    const uint8_t* ax = r.aux + (size_t)slot * kAuxBytes;
    const ChunkMeta* mp = reinterpret_cast<const ChunkMeta*>(ax + kAuxMeta);
    const float scale = mp->scale;
    const int planes = mp->planes, n_out = mp->n_out;
    const long long sum_x = mp->sum_x;
    const uint4* row0 =
        reinterpret_cast<const uint4*>(r.codes + (size_t)st * kStageBytes + (size_t)ra * kChunkRowBytes);
    const uint4* row1 = row0 + 32 * (kChunkRowBytes / 16);
    const uint4* pl = reinterpret_cast<const uint4*>(ax);
    float d0 = 0.f, d1 = 0.f;  // ungrouped: sum of T X over the chunk; grouped: the scaled sums
    if (grouped) {
      if (planes == 2) decode_unit_grouped<2>(row0, row1, pl, sw, mp, scale, gab0, gab1, d0, d1);
      else decode_unit_grouped<3>(row0, row1, pl, sw, mp, scale, gab0, gab1, d0, d1);
    } else if (planes == 2) {
      RowAcc<2> a0, a1;
      decode_unit<2>(row0, row1, pl, sw, a0, a1);
      d0 = finish_chunk2(a0, (int)sum_x);
      d1 = finish_chunk2(a1, (int)sum_x);
    } else {
      RowAcc<3> a0, a1;
      decode_unit<3>(row0, row1, pl, sw, a0, a1);
      d0 = finish_chunk3(a0, sum_x);
      d1 = finish_chunk3(a1, sum_x);
    }
    // outliers: T * v*x in fp32, the code of both rows read from the staged tile (byte col / 4 of
    // the row, in 16-byte granule (col / 64) ^ (row % 8) of the 128-byte swizzle; rows ra and ra + 32
    // share the swizzle phase)
    float o0 = 0.f, o1 = 0.f;
    if (n_out > 0) {
      const uint8_t* cb0 = reinterpret_cast<const uint8_t*>(row0);
      const uint8_t* cb1 = reinterpret_cast<const uint8_t*>(row1);
#pragma unroll 1
      for (int k = 0; k < n_out; ++k) {
        const int col = mp->out_col[k];
        const float xv = mp->out_val[k];
        const int off = ((((col >> 6) ^ sw) << 4) | ((col >> 2) & 15)), sh = 2 * (col & 3);
        float t0 = (float)(int)((cb0[off] >> sh) & 3u) - 1.f, t1 = (float)(int)((cb1[off] >> sh) & 3u) - 1.f;
        if (grouped) {  // scaled by the alpha of the outlier's group
          const int g = col >> 7;
          const uint32_t b0 = g == 0 ? gab0[0] : g == 1 ? gab0[1] : g == 2 ? gab0[2] : gab0[3];
          const uint32_t b1 = g == 0 ? gab1[0] : g == 1 ? gab1[1] : g == 2 ? gab1[2] : gab1[3];
          t0 *= h2f((uint16_t)(b0 & 0xffffu));
          t1 *= h2f((uint16_t)(b1 & 0xffffu));
        }
        o0 = fmaf(t0, xv, o0);
        o1 = fmaf(t1, xv, o1);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&r.empty_c[st]));  // codes and metadata no longer read
    yacc0 += grouped ? d0 + o0 : fmaf(d0, scale, o0);
    yacc1 += grouped ? d1 + o1 : fmaf(d1, scale, o1);

    // the previous unit's residual sums (into the tile they belong to), then its tile's epilogue
    if (pend >= 0) {
      float q0, q1;
      if (!take_residual(r, pend, pend_ph, ra, lane, q0, q1, status)) return;
      if (done) {
        dt.r0 += q0;
        dt.r1 += q1;
        tile_epilogue(r.tab[dt.p], dt, total, u0, u1, ra, et, status);
        done = false;
      } else {
        racc0 += q0;
        racc1 += q1;
      }
    }
    pend = slot;
    pend_ph = ph_a;
    if (c.ch == n_chunks - 1 || u == u1 - 1) {  // this CTA's part of tile c.t is decoded
      dt.y0 = yacc0;
      dt.y1 = yacc1;
      dt.r0 = racc0;
      dt.r1 = racc1;
      dt.al0 = al0;
      dt.al1 = al1;
      dt.p = c.p;
      dt.t = c.t;
      done = true;
      yacc0 = yacc1 = racc0 = racc1 = 0.f;
      need_alpha = true;
    }
    if (++st == r.S) {
      st = 0;
      ph_c ^= 1u;
    }
    if (++slot == kAuxSlots) {
      slot = 0;
      ph_a ^= 1u;
    }
    if (++c.ch == n_chunks) {
      c.ch = 0;
      if (++c.t == a.n_tiles) {
        c.t = 0;
        ++c.p;
      }
    }
  }
  // the last unit always ends a tile
  if (pend >= 0) {
    float q0, q1;
    if (!take_residual(r, pend, pend_ph, ra, lane, q0, q1, status)) return;
    if (done) {
      dt.r0 += q0;
      dt.r1 += q1;
      tile_epilogue(r.tab[dt.p], dt, total, u0, u1, ra, et, status);
    }
  }
}

template <int GM>
__global__ void __launch_bounds__(kThreads, 1)
    qtea_gemv_m1_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ GroupParams gp) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, formed by indexing (not through an integer) so that the compiler keeps
  // the shared address space and the hot loops use shared-memory loads
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int S = gp.n_stages;
  const int NP = gp.n_problems;
  const int u0 = gp.cta_u0[blockIdx.x], u1 = gp.cta_u0[blockIdx.x + 1];
  const int n_units = u1 - u0;

  Ring r;
  r.S = S;
  r.n_problems = NP;
  r.codes = smem;
  r.aux = smem + (size_t)S * kStageBytes;
  r.onehot = reinterpret_cast<float4*>(r.aux + (size_t)kAuxSlots * kAuxBytes);
  ProblemArgs* tab = reinterpret_cast<ProblemArgs*>(r.aux + (size_t)kAuxSlots * kAuxBytes +
                                                    (size_t)kHelperWarps * kOneHotBytes);
  r.tab = tab;
  r.full_c = reinterpret_cast<uint64_t*>(tab + kMaxProblems);
  r.empty_c = r.full_c + S;
  r.planes_a = r.empty_c + S;
  r.full_a = r.planes_a + kAuxSlots;
  r.empty_a = r.full_a + kAuxSlots;
  r.last_fill = reinterpret_cast<int*>(r.empty_a + kAuxSlots);

  // the problem table goes to shared memory in one step (every thread one word): reading it
  // from the parameter space field by field would be a chain of constant-cache misses
  {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(gp.prob);
    uint32_t* dst = reinterpret_cast<uint32_t*>(tab);
    const int words = NP * (int)(sizeof(ProblemArgs) / 4);
    for (int i = threadIdx.x; i < words; i += kThreads) dst[i] = src[i];
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_u32(&r.full_c[i]), 1);                // the producer's arrival with the TMA bytes
      mbar_init(smem_u32(&r.empty_c[i]), kConsumerWarps);  // one arrival per consumer warp
      r.last_fill[i] = 0;
    }
    for (int i = 0; i < kAuxSlots; ++i) {
      mbar_init(smem_u32(&r.planes_a[i]), 32);             // every lane of the helper
      mbar_init(smem_u32(&r.full_a[i]), 32);
      mbar_init(smem_u32(&r.empty_a[i]), kConsumerWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == kProducerWarp && lane < NP)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.m[lane])) : "memory");
  __syncthreads();

  // the first fill of every code stage: before the wait when the library owns the codes (no kernel
  // writes them after the layout is packed), after it when the caller does
  const bool pre_fill = gp.codes_after_wait == 0;
  if (pre_fill && warp == kProducerWarp && lane == 0) first_fills(maps, r, u0, n_units);
  // warm L2 with the lines of x and v that the first six units read (eight 128-byte lines of each
  // per 512-column chunk, one per helper lane): a prefetch reads no value into the SM, so the data
  // the units use is still read after the wait, from L2, where a preceding kernel's writes land
  if (warp >= kConsumerWarps && warp < kProducerWarp) {
    const int hl = (warp - kConsumerWarps) * 32 + lane, i = hl >> 4, l16 = hl & 15;
    if (i < n_units) {
      const UnitPos up = unit_pos(tab, NP, (long long)u0 + i);
      const ProblemArgs& pa = tab[up.p];
      const int col = up.ch * kChunkCols + (l16 & 7) * 64;  // 64 fp16 values per line
      if (col < pa.K)
        asm volatile("prefetch.global.L2 [%0];" ::"l"((l16 < 8 ? pa.x : pa.v) + col) : "memory");
    }
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (!pre_fill && warp == kProducerWarp && lane == 0) first_fills(maps, r, u0, n_units);

  if (warp < kConsumerWarps) consumer_role<GM>(r, gp.total_units, u0, u1, warp, lane, gp.status);
  else if (warp < kProducerWarp) helper_role(r, u0, n_units, warp - kConsumerWarps, lane, gp.status);
  else if (lane == 0) producer_role(maps, r, u0, n_units, gp.status);

  // no bulk copy may still be writing shared memory when the CTA exits (after a timeout the
  // consumers may not have waited for every fill)
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int s2 = 0; s2 < S; ++s2) {
      const int f = r.last_fill[s2];
      if (f > 0 && !mbar_wait(smem_u32(&r.full_c[s2]), (uint32_t)((f - 1) & 1), gp.status)) break;
    }
  }
}

}  // namespace

// Allow the kernel the largest dynamic shared memory the device grants next to its static
// shared memory; *dyn_max receives that size.
cudaError_t m1_configure(size_t smem_optin, size_t* dyn_max) {
  cudaFuncAttributes attr;
  cudaError_t e = cudaFuncGetAttributes(&attr, qtea_gemv_m1_kernel<1>);
  if (e != cudaSuccess) return e;
  const size_t dyn = smem_optin > attr.sharedSizeBytes ? smem_optin - attr.sharedSizeBytes : 0;
  *dyn_max = dyn;
  for (auto k : {qtea_gemv_m1_kernel<0>, qtea_gemv_m1_kernel<1>, qtea_gemv_m1_kernel<2>}) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// Programmatic stream serialisation lets this launch start while the previous kernel on the
// stream drains; the kernel waits for it (griddepcontrol.wait) before touching caller memory.
cudaError_t launch_m1(const TensorMaps& maps, const GroupParams& p, int grid, size_t smem, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // the variant holding only the decodes the launch's problems need (with or without scale groups,
  // or both): a smaller kernel, whose code stays in the instruction caches
  const int gm = p.n_grp == 0 ? 0 : p.n_grp == p.n_problems ? 2 : 1;
  return gm == 0 ? cudaLaunchKernelEx(&cfg, qtea_gemv_m1_kernel<0>, maps, p)
                 : gm == 2 ? cudaLaunchKernelEx(&cfg, qtea_gemv_m1_kernel<2>, maps, p)
                           : cudaLaunchKernelEx(&cfg, qtea_gemv_m1_kernel<1>, maps, p);
}

}  // namespace qtea
