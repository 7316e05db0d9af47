// Internal declarations shared by the host ABI and the kernels of the QTEA GEMV library.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "qtea.h"

namespace qtea {

// ---------------------------------------------------------------- batch-1 grouped stream-K kernel
// One CTA per SM: 8 consumer warps (each lane owns 2 rows of a 512-row tile) and 1 producer
// warp whose lane 0 drives the TMA ring. A unit of work is one (tile, chunk) pair of one
// problem: 512 rows x 512 columns = 512 x 128 bytes of 2-bit codes, fetched as two 2D TMA
// boxes of 256 rows with the 128-byte swizzle. One launch serves up to kMaxProblems
// independent GEMVs; their units form one sequence that is split evenly over the CTAs.
constexpr int kMaxProblems = 8;
constexpr int kMaxGrid = 1024;                                 // CTAs a launch may use
constexpr int kConsumerWarps = 8;
constexpr int kProducerWarp = kConsumerWarps;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kTileRows = 512;
constexpr int kBoxRows = 256;
constexpr int kChunkCols = 512;
constexpr int kChunkRowBytes = kChunkCols / 4;                 // 128
constexpr int kBoxBytes = kBoxRows * kChunkRowBytes;           // 32768
constexpr int kStageBytes = kTileRows * kChunkRowBytes;        // 65536
constexpr int kWordsPerChunk = kChunkCols / 16;                // 32 words of 16 codes
constexpr int kPlaneBytesPerWord = 48;                         // 4 groups x 3 byte planes x 4 bytes
constexpr int kPlaneBytesPerChunk = kWordsPerChunk * kPlaneBytesPerWord;  // 1536
constexpr int kMaxStages = 3;
constexpr int kMinStages = 2;
constexpr int kResidFloats = kConsumerWarps * 16 * 2 * 4;      // per-warp gather of residual sums

constexpr int kChunkSalCap = 64;                             // salient x values kept per staged chunk

struct ChunkMeta {
  float scale4;      // q / 4, q the fixed-point quantum of v*x in this chunk (a power of two)
  int c_lo, c_hi;    // salient entries whose column lies in the chunk
  int planes;        // byte planes of the chunk's fixed-point v*x: 3 (24-bit) or 2 (16-bit)
  long long sum_x;   // sum of the chunk's fixed-point v*x values
  long long pad2;
};

// One staged chunk: activation planes, metadata, and x at (up to kChunkSalCap of) the
// chunk's salient columns, in the order of the salient list.
constexpr int kSlotBytes = kPlaneBytesPerChunk + (int)sizeof(ChunkMeta) + kChunkSalCap * 4;  // 1824

struct ProblemArgs {
  const uint16_t* x;        // [K] (M = 1)
  const uint16_t* alpha;    // [N]
  const uint16_t* v;        // [K]
  const int32_t* sal;       // [s]
  const uint16_t* rvals;    // [N/4][s]
  const uint8_t* ridx;      // [N/4][ceil(s/4)]
  float* y;                 // [N]
  float* ws;                // [grid][2][kTileRows] partial sums of split tiles
  unsigned* counters;       // [n_tiles][kConsumerWarps], zero between calls
  int N, K, s, n_tiles, n_chunks;
  int act_bits;             // 24: v*x in 24-bit fixed point; 16: 16-bit where a chunk allows it
  long long unit_begin;     // first global unit of this problem
};

struct TensorMaps {
  CUtensorMap m[kMaxProblems];
};

struct GroupParams {
  ProblemArgs prob[kMaxProblems];
  int n_problems, n_stages;
  int* status;              // device status word (the first layout's)
  long long total_units;
  int cta_u0[kMaxGrid + 1]; // first unit of every CTA (balanced split), cta_u0[grid] = total
};

// First unit of CTA b in a balanced split of `total` units over `grid` CTAs.
__host__ __device__ inline long long unit_begin_of(int b, long long total, int grid) {
  return (long long)b * total / grid;
}

// Per-problem staging of one CTA: the cyclic range of chunks its units touch.
struct StageSlot {
  int p;         // problem index
  int ch_start;  // first chunk (cyclic range)
  int n_ch;      // number of chunks staged
  int s;         // salient count of the problem
  int chunks;    // byte offset of n_ch chunk slots of kSlotBytes
  int salc;      // byte offset of the clamped salient column indices (s ints)
  int first_unit;  // first unit of this problem in the CTA's range
  int pad;
};

// Shared-memory plan of the CTA whose units are [u0, u1). Identical on host (for the launch
// size) and device.
__host__ __device__ inline size_t cta_smem_plan(const ProblemArgs* prob, int n_problems, int n_stages, int u0, int u1,
                                                StageSlot* slots, int* n_slots, size_t* misc_off) {
  size_t off = (size_t)n_stages * kStageBytes;  // ring first, at the 1024-aligned base
  int ns = 0;
  for (int p = 0; p < n_problems; ++p) {
    const ProblemArgs& a = prob[p];
    const int pb = (int)a.unit_begin, pe = (int)a.unit_begin + a.n_tiles * a.n_chunks;
    const int lo = u0 > pb ? u0 : pb, hi = u1 < pe ? u1 : pe;
    if (lo >= hi) continue;
    StageSlot sl;
    sl.p = p;
    sl.ch_start = (lo - pb) % a.n_chunks;
    const int n = hi - lo;
    sl.n_ch = n >= a.n_chunks ? a.n_chunks : n;
    sl.s = a.s;
    sl.first_unit = lo;
    sl.pad = 0;
    off = (off + 15) & ~(size_t)15;
    sl.chunks = (int)off;
    off += (size_t)sl.n_ch * kSlotBytes;
    sl.salc = (int)off;
    off += (size_t)(a.s > 0 ? a.s : 1) * sizeof(int);
    if (slots) slots[ns] = sl;
    ++ns;
  }
  off = (off + 15) & ~(size_t)15;
  if (misc_off) *misc_off = off;
  // misc: residual gather floats, staging table, barriers (ring full/empty)
  off += (size_t)kResidFloats * sizeof(float);
  off += (size_t)kMaxProblems * sizeof(StageSlot);
  off += (size_t)2 * n_stages * sizeof(unsigned long long);
  if (n_slots) *n_slots = ns;
  return off + 1024;  // slack to align the dynamic smem base to 1024 bytes
}

// ---------------------------------------------------------------- generic kernel (any M)
struct GenericParams {
  const uint16_t* x;        // [M][K]
  const uint8_t* packed;    // [N][K_pad/4]
  const uint16_t* alpha;    // [N]
  const uint16_t* v;        // [K]
  const int32_t* sal;       // [s]
  const uint16_t* rvals;    // [N/4][s]
  const uint8_t* ridx;      // [N/4][ceil(s/4)]
  float* y;                 // [M][N]
  int M, N, K, K_pad, s;
};

cudaError_t launch_m1(const TensorMaps& maps, const GroupParams& p, int grid, size_t smem, cudaStream_t st);
cudaError_t m1_configure(size_t smem_optin, size_t* dyn_max);
cudaError_t launch_generic(const GenericParams& p, cudaStream_t st);
cudaError_t launch_pack(const int8_t* codes, int N, int K, int K_pad, uint32_t* packed, int* bad_flag,
                        cudaStream_t st);

}  // namespace qtea

struct qtea_layout {
  int N, K, K_pad, group_size, n_salient, format;
  size_t packed_bytes;
  uint8_t* packed;
  int device;
  int sm_count;
  size_t smem_optin;
  // batch-1 kernel resources
  bool m1_ok;
  int act_bits;          // activation precision of batch-1 calls: 24 (default) or 16
  int n_tiles, n_chunks;
  float* workspace;      // [sm_count][2][kTileRows]
  unsigned* counters;    // [n_tiles][kConsumerWarps]
  int* status;
  CUtensorMap tmap;
};
