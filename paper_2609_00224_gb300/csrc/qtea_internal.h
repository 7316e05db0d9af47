// Internal declarations shared by the host ABI and the kernels of the QTEA GEMV library.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "qtea.h"

namespace qtea {

// ---------------------------------------------------------------- batch-1 grouped stream-K kernel
// One CTA per SM: 8 consumer warps decode (each lane owns 2 rows of a 512-row tile), 3 helper
// warps stage activations and residual sums, 1 producer warp drives the TMA. A unit of work is
// one (tile, chunk) pair of one problem: 512 rows x 512 columns = 512 x 128 bytes of 2-bit codes,
// fetched by TMA as two 2D boxes of 256 rows with the 128-byte swizzle into a code stage. Its
// auxiliary slot (in a deeper ring of its own) holds the chunk's fixed-point v*x planes and the
// unit's share of the residual as one sum per row. One launch serves up to kMaxProblems
// independent GEMVs; their units form one sequence that is split evenly over the CTAs.
constexpr int kMaxProblems = 8;
constexpr int kMaxGrid = 1024;                                 // CTAs a launch may use
constexpr int kConsumerWarps = 8;
constexpr int kHelperWarps = 3;                                // activation / residual staging
constexpr int kProducerWarp = kConsumerWarps + kHelperWarps;  // TMA issue
constexpr int kThreads = (kProducerWarp + 1) * 32;             // 384
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
constexpr int kAuxSlots = 2 * kHelperWarps;                    // each helper owns two slots
constexpr int kResBlock = 8;                                   // salient entries per residual block

// Elements of a chunk's v*x at least 16 times larger than every other element (found in up to
// kOutlierRounds rounds) are taken out of the fixed-point planes, up to kMaxOutliers of them, and
// added exactly in fp32 (T * v*x per row, the code read from the staged tile).
constexpr int kMaxOutliers = 16;
constexpr int kOutlierRounds = 4;

struct ChunkMeta {  // 160 bytes
  float scale;       // q, the fixed-point quantum of v*x in this chunk (a power of two)
  int planes;        // byte planes of the chunk's fixed-point v*x: 3 (24-bit) or 2 (16-bit)
  long long sum_x;   // sum of the chunk's fixed-point v*x values (outliers excluded)
  int n_out;         // outliers of the chunk (0 .. kMaxOutliers)
  int pad[3];
  uint16_t out_col[kMaxOutliers];  // their columns within the chunk
  float out_val[kMaxOutliers];     // their v*x, exact
  int gsum_x[4];     // scale groups: the fixed-point v*x summed per 128-column group
  float gsx[4];      // scale groups with beta: x summed per 128-column group
};

// Auxiliary slot: planes [32 words][48 bytes], metadata, residual sums [512 rows].
constexpr int kAuxMeta = kPlaneBytesPerChunk;
constexpr int kAuxRes = kAuxMeta + (int)sizeof(ChunkMeta);
constexpr int kAuxBytes = kAuxRes + kTileRows * (int)sizeof(float);  // 3744
// Per helper: x at one residual block's 8 entries spread over the 4 positions of a group,
// T[entry][position] = x * one-hot(position), so that an entry adds with 4 FMAs and no selects.
constexpr int kOneHotBytes = kResBlock * 4 * 16;               // 512

struct ProblemArgs {
  const uint16_t* x;        // [K] (M = 1)
  const uint16_t* alpha;    // [N] alpha, or with scale groups [N][G] alpha or [N][G][2] (alpha, beta)
  const uint16_t* v;        // [K]
  const int32_t* sal;       // [s]
  const uint16_t* rvals;    // [N/4][s]
  const uint8_t* ridx;      // [N/4][ceil(s/4)]
  float* y;                 // [N]
  float* ws;                // [grid][2][kTileRows] partial rows of split tiles (slot 0 used), zero between calls
  unsigned* counters;       // [n_tiles][kConsumerWarps], zero; not used by the batch-1 kernels
  int N, K, s, n_tiles, n_chunks;
  int act_bits;             // 24: v*x in 24-bit fixed point; 16: 16-bit where a chunk allows it
  int vec_xv;               // x and v are 16-byte aligned (vector loads)
  int vec_res;              // s % 8 == 0 and rvals 16-byte / ridx 2-byte aligned (vector loads)
  int gflags;               // kScaleGroups | kScaleBias | kScaleVec (one int: the struct stays 128 bytes,
                            // which keeps the kernel's copies of it out of local memory)
  int G, gdiv;              // scale groups per row; 128-column groups per scale group
  long long unit_begin;     // first global unit of this problem
};

// ProblemArgs::gflags: alpha (and beta) applied per 128-column group inside the decode; beta
// present; a row's four groups of a chunk are one aligned 16-byte (8 without beta) load.
constexpr int kScaleGroups = 1, kScaleBias = 2, kScaleVec = 4;
static_assert(sizeof(ProblemArgs) <= 128, "larger problem records spill the batch-1 kernel's copies");

struct TensorMaps {
  CUtensorMap m[kMaxProblems];
};

struct GroupParams {
  ProblemArgs prob[kMaxProblems];
  int n_problems, n_stages;
  int n_grp;                // problems with scale groups (the kernel variants: none, some, all)
  int codes_after_wait;     // the codes belong to the caller: no code fill before the grid dependency wait
  int* status;              // device status word (the first layout's)
  long long total_units;
  int cta_u0[kMaxGrid + 1]; // first unit of every CTA (balanced split), cta_u0[grid] = total
};

// First unit of CTA b in a balanced split of `total` units over `grid` CTAs.
__host__ __device__ inline long long unit_begin_of(int b, long long total, int grid) {
  return (long long)b * total / grid;
}

// Dynamic shared memory of the batch-1 kernel with S code stages: codes, auxiliary slots, the
// helpers' one-hot tables, the problem table, the barriers (code stages: full, empty; auxiliary slots: planes written, residual
// written, empty), the fills issued per code stage (for the drain), and 1024 bytes of slack.
__host__ __device__ constexpr size_t m1_smem_bytes(int S) {
  return (size_t)S * kStageBytes + (size_t)kAuxSlots * kAuxBytes + (size_t)kHelperWarps * kOneHotBytes +
         (size_t)kMaxProblems * sizeof(ProblemArgs) +
         (size_t)(2 * S + 3 * kAuxSlots) * sizeof(unsigned long long) + (size_t)kMaxStages * sizeof(int) + 1024;
}

// ---------------------------------------------------------------- row-resident batch-1 kernel (small groups)
// For small groups: every CTA owns whole rows (up to kRowsMaxRows, in 8-row blocks; one or two CTAs
// per SM) of one problem, so no partial sums cross CTAs. Its codes arrive by TMA before the grid
// dependency wait, one barrier per 512-column chunk (8-row boxes of 128 bytes, 128-byte swizzle);
// warp w stages the planes of chunks w, w + 8, ... and decodes each for all of the CTA's rows.
// Narrow launches (K <= 4096: one chunk per warp, at most kRowsMaxSalient salient columns) may put
// two CTAs on an SM; wide ones (up to kRowsMaxChunks chunks, kRowsMaxSalientWide salient columns)
// one, with the registers that leaves for the next chunk's x and v and every residual operand.
constexpr int kRowsWarps = 8;
constexpr int kRowsThreads = kRowsWarps * 32;                  // 256
constexpr int kRowsMaxRows = 32;                               // one row per lane
constexpr int kRowsBoxRows = 8;
constexpr int kRowsSlotBytes = 1792;                           // planes + ChunkMeta of one chunk, per warp
constexpr int kRowsMaxSalient = 256;                           // narrow: salient columns (half of them in registers)
// wide: 512-column chunks (K <= 8192), two per warp at most. Measured single calls: 1024 x 5120
// 8.4 -> 5.5 us and 1024 x 8192 8.5 -> 6.2 us against the stream-K kernel, but 4096 x 14336 (28
// chunks, 3.5 per warp) 10.2 -> 11.7 us: a warp's chunks are staged and decoded one after another.
constexpr int kRowsMaxChunks = 16;
constexpr int kRowsMaxSalientWide = 512;                       // wide: salient columns, all in registers

struct RowsParams {
  ProblemArgs prob[kMaxProblems];   // as for the stream-K kernel (ws, counters, n_tiles, unit_begin unused)
  int cta_begin[kMaxProblems + 1];  // CTAs of problem p: [cta_begin[p], cta_begin[p + 1])
  int rows_cap;                     // rows of a CTA's buffer per chunk (multiple of 8, at most kRowsMaxRows)
  int n_chunks_max;                 // over the problems: shared-memory size
  int n_problems;
  int kparts;                       // lanes per row of every CTA (1, 2 or 4), or 0: each CTA by its rows
  int wide;                         // 1: some problem has more than kRowsWarps chunks or more than
                                    // kRowsMaxSalient salient columns (one CTA per SM)
  int* status;                      // device status word (the first layout's)
};

// Dynamic shared memory of the row-resident kernel (offsets from the 1024-byte aligned base):
// codes [n_chunks_max][rows_cap][128], the warps' plane slots, their partial row sums, the
// residual per row, the CTA's problem record, the code barriers, and 1024 bytes of slack.
struct RowsSmem {
  size_t slots, dec, res, args, bars, total;
};
__host__ __device__ inline RowsSmem rows_smem_layout(int rows_cap, int n_chunks_max) {
  RowsSmem o;
  o.slots = (size_t)n_chunks_max * rows_cap * kChunkRowBytes;
  o.dec = o.slots + (size_t)kRowsWarps * kRowsSlotBytes;
  o.res = o.dec + (size_t)kRowsWarps * kRowsMaxRows * sizeof(float);
  o.args = o.res + (size_t)kRowsMaxRows * sizeof(float);
  o.bars = o.args + sizeof(ProblemArgs);
  o.total = o.bars + (size_t)n_chunks_max * sizeof(unsigned long long) + 1024;
  return o;
}

cudaError_t rows_configure(size_t smem_optin);
cudaError_t launch_rows(const TensorMaps& maps, const RowsParams& p, int grid, size_t smem, cudaStream_t st);

// ---------------------------------------------------------------- low-batch tensor-core kernel (2 <= M <= 16)
constexpr int kMaxStagesMb = 6;
constexpr int kMinStagesMb = 2;
constexpr int kMbTileRows = 256;                               // rows of a unit (one TMA box)
constexpr int kMbVBytes = 1024;                                // v of a chunk in fragment order
constexpr int kMbSxBytes = 256;                                // sum of x per 128-column group and batch row [4][16] fp32
constexpr int kMbChunkHead = kMbVBytes + kMbSxBytes;           // the x blocks start here
constexpr int kMbXTileBytes = 8192;                            // x of a chunk, 8 batch rows, fragment order
constexpr int kMbChunkWsBytes = kMbChunkHead + 2 * kMbXTileBytes;  // 17664 per 512-column chunk
// Split encoding (M <= 8): the chunk head holds, instead of v, the chunk's fold factor 2^(-E-1)
// (fp32) at kMbHlF; the blocks hold B = the exact fp16 (hi, lo) split of v*x * 2^E (see the
// kernel's header).
constexpr int kMbHlF = 0;
// Scratch of the chunk build: x [16][512] and v [512] fp16, then eight warp maxima.
constexpr int kMbPrepScratch = 16 * kChunkCols * 2 + kChunkCols * 2 + 64;
// n8 tiles of the B operand and the encoding for batch size M: the split encoding (v*x as fp16 hi
// and lo in two columns per batch row, one tile) for M <= 4; 2T*v with B = x for 5 <= M <= 16, one
// tile up to M = 8 and two up to 16. (Measured on the Qwen3-14B layer: the split encoding in two
// tiles at M = 8 took 50.5 us against 42.8 for 2T*v in one.)
__host__ __device__ constexpr bool mb_split(int M) { return M <= 4; }
__host__ __device__ constexpr int mb_mt(int M) { return M <= 8 ? 1 : 2; }
constexpr int kMbAbBytes = 256 * 16;                           // alpha (and beta) of a unit's rows, 8 fp16 per row

// One shared-memory stage of the low-batch kernel: codes [256 rows][128 bytes], the chunk's v block,
// group sums of x and MT x blocks, with scale groups the unit's alpha (and beta), rounded to 1024
// bytes (the 128-byte swizzle of the next stage's codes).
__host__ __device__ constexpr int mb_stage_bytes(int mt, bool grp) {
  return (kMbTileRows * kChunkRowBytes + kMbChunkHead + mt * kMbXTileBytes + (grp ? kMbAbBytes : 0) + 1023) / 1024 *
         1024;
}

// Prep kernel: v and x of every 512-column chunk in fragment order, and the residual (Eq. 11) of
// every 256-row tile in the consumers' accumulator order, for every problem of a group in one launch.
constexpr int kMbResEntries = 256;  // salient entries staged per pass of a residual block

// How a problem's residual (Eq. 11) is computed: not at all (s = 0), by the main kernel's helper
// warps from bulk copies, or per tile by the prep kernel.
enum MbResMode { kMbResNone = 0, kMbResHelpers = 1, kMbResPrep = 2 };

struct MbPrepProblem {
  const uint16_t* x;        // [M][K]
  const uint16_t* v;        // [K]
  const int32_t* sal;       // [s]
  const uint16_t* rvals;    // [N/4][s]
  const uint8_t* ridx;      // [N/4][ceil(s/4)]
  uint8_t* ws;              // [n_chunks][kMbChunkWsBytes]
  float* yres;              // kMbResPrep: [n_tiles][256 threads][4 kMbBlocks MT] residual in accumulator order
  uint16_t* xs;             // kMbResHelpers: x at the salient columns [16][s16]
  int N, K, s, s16, n_chunks, n_tiles;
  int res_mode;
  int native;               // kMbResPrep: residual staged as stored (16-byte vector loads), else in passes
  int block_begin;          // first block of this problem in the launch
};

struct MbPrepGroup {
  MbPrepProblem prob[kMaxProblems];
  int n_problems, M, mt, n_blocks;
  int split;                // mb_split(M): the split encoding's chunks
  size_t smem;              // dynamic shared memory of a block
};

constexpr int kMbBlocks = 2;                                   // 16-row blocks per consumer warp
constexpr int kMbConsumerWarps = kMbTileRows / 16 / kMbBlocks;  // 8
constexpr int kMbHelperWarps = 4;                              // residual of the tiles a CTA starts

// One problem of a grouped low-batch launch; units (tile of 256 rows, chunk of 512 columns) of all
// problems form one sequence split evenly over the CTAs, as in the batch-1 kernel.
struct MbProblemArgs {
  const uint16_t* alpha;    // [N]
  const uint8_t* ws;        // the prep kernel's chunks
  const float* yres;        // kMbResPrep: the prep kernel's residual per tile
  const uint16_t* rvals;    // kMbResHelpers: [N/4][s], 16-byte aligned
  const uint8_t* ridx;      // kMbResHelpers: [N/4][ceil(s/4)], 16-byte aligned
  const uint16_t* xs;       // kMbResHelpers: the prep kernel's x at the salient columns [16][s16]
  float* y;                 // [M][N]
  float* part;              // [grid][2][256 threads][4 kMbBlocks MT] partial rows of split tiles (slot 0 used), zero between calls
  unsigned* counters;       // [n_tiles][kMbConsumerWarps], zero; not used by the kernel
  int N, n_tiles, n_chunks, s, s16, res_mode;
  int res_passes;           // kMbResHelpers: a tile's row groups are staged in 1, 2 or 4 passes
  int bias;                 // scale groups: row_scale holds (alpha, beta) pairs
  int fp8;                  // kMbResHelpers: residual values in FP8 E4M3 (one byte each)
  long long unit_begin;
};

struct MbGroupParams {
  MbProblemArgs prob[kMaxProblems];
  MbPrepGroup prep;         // fused: the prep work, done by the main kernel's CTAs before a grid barrier
  int fused;
  unsigned long long* gbar; // fused: grid barrier counter (monotonic), target below
  unsigned long long gbar_target;
  int n_problems, n_stages, M;
  int split;                // mb_split(M)
  int res_stage_bytes;      // the helpers' staging buffer (and the fused prep's scratch)
  int* status;              // device status word (the first layout's)
  long long total_units;
  int cta_u0[kMaxGrid + 1];
};

// Partial-row slots of the low-batch kernel per layout: [sm_count][2][256 threads][16] floats.
constexpr size_t kMbPartFloatsPerCta = 2 * 256 * 16;
// Residual of one 256-row tile in accumulator order: [256 threads][16] floats.
constexpr size_t kMbResFloatsPerTile = 256 * 16;

// Helpers' staging of one pass over a tile's residual: the values (2 bytes each, or 1 in FP8) and
// position bytes of 64 / passes row groups as stored, and x at the salient columns [16][s16].
__host__ __device__ inline size_t mb_res_stage_bytes(int s, int passes, bool fp8) {
  const size_t g = (size_t)(kMbTileRows / 4 / passes), rs = (size_t)((s + 3) / 4), s16 = (size_t)((s + 15) / 16 * 16);
  return ((g * s * (fp8 ? 1 : 2) + 15) & ~(size_t)15) + ((g * rs + 15) & ~(size_t)15) + 16 * s16 * 2;
}

// Shared memory of the low-batch kernel (offsets from the 1024-byte aligned base).
struct MbSmem {
  size_t tab, rslot, rstage, bars, last_fill, total;
};
__host__ __device__ inline MbSmem mb_smem_layout(int S, int mt, bool grp, int res_stage_bytes) {
  MbSmem o;
  o.tab = (size_t)S * mb_stage_bytes(mt, grp);
  o.rslot = (o.tab + kMaxProblems * sizeof(MbProblemArgs) + 127) & ~(size_t)127;
  o.rstage = (o.rslot + (size_t)2 * 256 * 8 * mt * sizeof(float) + 127) & ~(size_t)127;
  o.bars = (o.rstage + (size_t)res_stage_bytes + 127) & ~(size_t)127;
  o.last_fill = o.bars + (size_t)(2 * S + 5) * 8;  // full, empty [S]; res_full, res_empty [2]; staged
  o.total = o.last_fill + (size_t)kMaxStagesMb * sizeof(int) + 1024;
  return o;
}

size_t mb_smem_bytes(int S, int M, bool grp, int res_stage_bytes);
cudaError_t mb_configure(size_t smem_optin, size_t* dyn_max);
size_t mb_prep_smem_bytes(int s, bool native);
cudaError_t mb_prep_configure(size_t smem_optin);
cudaError_t launch_mb_prep(const MbPrepGroup& g, cudaStream_t st);
// Scale groups (grp): alpha, or (alpha, beta) pairs, per row and 128-column group, loaded per unit
// by TMA through `ab_maps` (row_scale as [N][G] or [N][2G] fp16, box 8 x 256).
cudaError_t launch_mb(const TensorMaps& maps, const TensorMaps& ab_maps, const MbGroupParams& p, bool grp, int grid,
                      size_t smem, cudaStream_t st);

// ---------------------------------------------------------------- table-lookup kernel (base-3, M = 1)
// The paper's decode (Sec. 3.5, Appendix A): per chunk of 8 blocks of 128 columns (208 code bytes
// per row) a sign-symmetric table of 122 fp32 dot products per code byte, in shared memory; 16 warps
// of 32 rows each make a 512-row tile.
constexpr int kLutWarps = 16;
constexpr int kLutThreads = kLutWarps * 32;
constexpr int kLutTileRows = kLutWarps * 32;                   // 512
constexpr int kLutBlocks = 8;                                  // 128-column blocks per chunk
constexpr int kLutCols = kLutBlocks * 128;                     // 1024
constexpr int kLutPacks = kLutBlocks * 26;                     // 208 code bytes per row and chunk
constexpr int kLutLanes = kLutPacks / 8;                       // 26 lanes of 8 code bytes
constexpr int kLutHalf = 122;                                  // entries of a half table
constexpr int kLutStride = 224;                                // floats per table row (7 x 32 banks)
constexpr int kLutMaxEntries = 1040;                           // salient entries a chunk may take
constexpr int kLutResBatch = 32;                               // salient entries per residual batch
// table, v*x of the chunk, x at the chunk's salient columns, the blocks' sums of x, (alpha, beta) of
// the tile's rows and the chunk's blocks (scale groups)
constexpr size_t kLutSmemBytes =
    (size_t)(kLutHalf * kLutStride + kLutCols + kLutMaxEntries + kLutBlocks + kLutTileRows * kLutBlocks) * 4;

struct LutProblem {
  const uint16_t* x;        // [K]
  const uint8_t* packed;    // [N][row_bytes] base-3
  const uint16_t* scales;   // [N] alpha, or with groups [N][G] alpha or [N][G][2] (alpha, beta)
  const uint16_t* v;        // [K]
  const int32_t* sal;       // [s]
  const void* rvals;        // [N/4][s] fp16, or FP8 E4M3 bytes
  const uint8_t* ridx;      // [N/4][ceil(s/4)]
  float* y;                 // [N]
  float* ws;                // [grid][2][kLutTileRows] partial rows of split tiles
  unsigned* counters;       // [n_tiles][kLutWarps], zero between calls
  int N, K, s, row_bytes, n_blocks, n_tiles, n_chunks;
  int fp8;                  // residual values in FP8 E4M3
  int aligned8;             // rows start on 8-byte boundaries (8-byte code loads)
  int G, bias;              // scale groups per row (the launch's variant when grouped), beta present
  int gdiv;                 // 128-column blocks per scale group (1, or all of them with one group)
  long long unit_begin;     // first unit of this problem in the launch
};

struct LutParams {
  LutProblem prob[kMaxProblems];
  int n_problems;
  long long total_units;
  int cta_u0[kMaxGrid + 1];
};

cudaError_t lut_configure(size_t smem_optin);
cudaError_t launch_lut(const LutParams& p, bool grouped, int grid, cudaStream_t st);

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

// Layouts in the paper's own storage (base-3 codes, scale groups of 128 columns, beta, FP8
// residual values): one warp per output row, any batch.
struct PaperParams {
  const uint16_t* x;        // [M][K]
  const uint8_t* packed;    // [N][row_bytes]: 2-bit (K_pad/4 bytes per row) or base-3 (26 per 128 columns)
  const uint16_t* scales;   // [N][G] alpha, or [N][G][2] (alpha, beta) with bias
  const uint16_t* v;        // [K]
  const int32_t* sal;       // [s]
  const void* rvals;        // [N/4][s] fp16, or FP8 E4M3 bytes with residual_fp8
  const uint8_t* ridx;      // [N/4][ceil(s/4)]
  float* y;                 // [M][N]
  int M, N, K, s, G, group_size, row_bytes, format, bias, residual_fp8;
  int staged_ok, sm_count;   // the staged-activation kernel is configured; SMs of the device
  size_t smem_optin, smem_per_sm;
};

// The quantizer's per-layer steps (qtea_quant.cu).
struct QuantArgs {
  const float* W;           // [N][K]
  const float* h;           // [K] diag(H)
  int N, K, group, s, bias, fit_iters, rescale_iters;
  int8_t* codes;            // [N][K]
  uint16_t* row_scale;      // [N][G] alpha, or [N][G][2] (alpha, beta)
  uint16_t* col_scale;      // [K] v
  int32_t* sal;             // [s]
  uint16_t* rvals;          // [N/4][s]
  uint8_t* ridx;            // [N/4][ceil(s/4)]
};

cudaError_t launch_quantize(const QuantArgs& a, cudaStream_t st);
// Up to eight base-3 problems of one batch size in one launch; work[q] = sum over earlier problems of
// rows x 128-column blocks.
struct B3Group {
  PaperParams prob[8];
  long long work[9];
  int n;
};

cudaError_t launch_paper(const PaperParams& p, cudaStream_t st);
cudaError_t launch_b3(const B3Group& g, cudaStream_t st);
bool b3_eligible(const PaperParams& p);
cudaError_t paper_configure(size_t smem_optin);
cudaError_t launch_pack_base3(const int8_t* codes, int N, int K, uint8_t* packed, int* bad_flag, cudaStream_t st);
cudaError_t launch_m1(const TensorMaps& maps, const GroupParams& p, int grid, size_t smem, cudaStream_t st);
// Sec. 3.5's salient bitmap (column j at bit j % 32 of word j / 32) and the ascending index list.
cudaError_t launch_bitmap_to_index(const uint32_t* bitmap, int K, int32_t* idx, int max_s, int* count,
                                   cudaStream_t st);
cudaError_t launch_index_to_bitmap(const int32_t* idx, int s, int K, uint32_t* bitmap, int* bad, cudaStream_t st);
cudaError_t m1_configure(size_t smem_optin, size_t* dyn_max);
cudaError_t launch_generic(const GenericParams& p, cudaStream_t st);
cudaError_t launch_pack(const int8_t* codes, int N, int K, int K_pad, uint32_t* packed, int* bad_flag,
                        cudaStream_t st);


#ifdef __CUDACC__
#include <cuda_fp16.h>

// ---------------------------------------------------------------- device helpers shared by the kernels
// Bounded waits give up after this long (then the kernel records QTEA_ERR_TIMEOUT and its role stops).
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

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

// One potentially blocking test of the phase with the given parity (the thread may be suspended
// for a system-dependent time until the phase completes).
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait until the phase with the given parity has completed; false after kWaitLimitNs, with
// QTEA_ERR_TIMEOUT recorded in *status.
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

// Tiled 2D TMA load of one box at (x, y) into shared memory, completing on mbarrier `bar`.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// An L2 cache policy that marks lines as the first to evict: for data streamed once per call (the
// packed codes), so that they do not push out of L2 what the next calls read again.
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// tma_load_2d with an L2 cache policy for the lines it reads.
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar,
                                                 uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(pol)
      : "memory");
}

__device__ __forceinline__ float h2f(uint16_t b) { return __half2float(__ushort_as_half(b)); }

// OFP8 E4M3 (the paper's residual format, Sec. 4.1): bias 7, subnormals m * 2^-9, S.1111.111 is
// NaN, no infinity; every value exact in fp32.
__device__ __forceinline__ float e4m3_to_float(uint32_t b) {
  const uint32_t e = (b >> 3) & 15u, m = b & 7u;
  float mag;
  if (e == 15u && m == 7u) mag = __int_as_float(0x7fc00000);
  else if (e == 0u) mag = (float)m * 0.001953125f;
  else mag = __int_as_float((int)((e + 120u) << 23 | m << 20));
  return (b & 0x80u) ? -mag : mag;
}
#endif  // __CUDACC__

}  // namespace qtea

struct qtea_layout {
  int N, K, K_pad, group_size, n_salient, format;
  int options;           // QTEA_OPT_* flags (qtea_set_layout_options)
  int row_bytes;         // packed bytes per row
  size_t packed_bytes;
  uint8_t* packed;
  int device;
  int sm_count;
  size_t smem_optin;
  size_t smem_per_sm;
  bool paper_staged_ok;  // the paper-storage kernel with staged activations is configured
  // batch-1 kernel resources
  bool m1_ok;
  int act_bits;          // activation precision of batch-1 calls: 24 (default) or 16
  int n_tiles, n_chunks;
  float* workspace;      // [sm_count][2][kTileRows]
  unsigned* counters;    // [n_tiles][kConsumerWarps]
  int* status;
  CUtensorMap tmap;
  bool rows_ok;          // the row-resident kernel is configured and tmap8 encoded
  CUtensorMap tmap8;     // the codes in boxes of 8 rows x 128 bytes (row-resident kernel)
  size_t rows_smem_optin;  // dynamic shared memory the row-resident kernel may use
  // low-batch kernel resources
  bool mb_ok;
  size_t mb_smem_optin;
  size_t prep_smem_optin;  // dynamic shared memory the prep kernel may use
  unsigned long long* mb_gbar;                // grid barrier counter of fused low-batch launches
  mutable unsigned long long mb_gbar_next;    // its value after the last launch issued (host side)
  uint8_t* mb_ws;        // [n_chunks][kMbChunkWsBytes] v and x in fragment order, then the residual
                         // of every 256-row tile [n_tiles][kMbResFloatsPerTile]
  float* mb_part;        // [sm_count][kMbPartFloatsPerCta] partial rows of split tiles
  unsigned* mb_counters; // [n_tiles of 256 rows][kMbConsumerWarps]
  // table-lookup kernel resources (base-3 layouts)
  bool lut_ok;
  float* lut_ws;         // [sm_count][2][kLutTileRows]
  unsigned* lut_counters;  // [n_tiles of 512 rows][kLutWarps]
};
