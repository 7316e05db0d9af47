// Host side of the C ABI declared in include/qtea.h: argument validation, layout ownership,
// launch planning and dispatch. No computation happens on the host.
#include <cudaTypedefs.h>

#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>

#include "qtea_internal.h"

using namespace qtea;

namespace {

// Below this many input columns the 16-bit activation mode is not used: with few nonzeros per
// row its rounding errors average out less.
constexpr int kMinK16 = 1024;

int round_up(int a, int b) { return (a + b - 1) / b * b; }

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

PFN_cuTensorMapEncodeTiled_v12000 get_encode_tiled() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

void release(qtea_layout* l) {
  if (!l) return;
  if (l->packed) cudaFree(l->packed);
  if (l->workspace) cudaFree(l->workspace);
  if (l->counters) cudaFree(l->counters);
  if (l->status) cudaFree(l->status);
  if (l->mb_ws) cudaFree(l->mb_ws);
  if (l->mb_gbar) cudaFree(l->mb_gbar);
  if (l->mb_part) cudaFree(l->mb_part);
  if (l->mb_counters) cudaFree(l->mb_counters);
  if (l->lut_ws) cudaFree(l->lut_ws);
  if (l->lut_counters) cudaFree(l->lut_counters);
  delete l;
}

// Resources of the batch-1 kernel for one layout: its TMA descriptor (512-row x 512-column
// units, two 256-row boxes each) and the split-tile workspace.
int plan_m1(qtea_layout* l, const cudaDeviceProp& prop) {
  l->m1_ok = false;
  l->sm_count = prop.multiProcessorCount;
  l->smem_optin = prop.sharedMemPerBlockOptin;
  if (l->N == 0 || l->K == 0) return QTEA_OK;
  l->n_tiles = (l->N + kTileRows - 1) / kTileRows;
  l->n_chunks = (l->K_pad + kChunkCols - 1) / kChunkCols;
  PFN_cuTensorMapEncodeTiled_v12000 encode = get_encode_tiled();
  if (!encode) return QTEA_OK;
  cuuint64_t dims[2] = {(cuuint64_t)(l->K_pad / 4), (cuuint64_t)l->N};
  cuuint64_t strides[1] = {(cuuint64_t)(l->K_pad / 4)};
  cuuint32_t box[2] = {(cuuint32_t)kChunkRowBytes, (cuuint32_t)kBoxRows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = encode(&l->tmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, l->packed, dims, strides, box, estr,
                      CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return QTEA_OK;
  {
    // the row-resident kernel: the same codes in boxes of 8 rows
    cuuint32_t box8[2] = {(cuuint32_t)kChunkRowBytes, (cuuint32_t)kRowsBoxRows};
    l->rows_ok = encode(&l->tmap8, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, l->packed, dims, strides, box8, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS &&
                 rows_configure(prop.sharedMemPerBlockOptin) == cudaSuccess;
    if (!l->rows_ok) cudaGetLastError();
    l->rows_smem_optin = prop.sharedMemPerBlockOptin;
  }
  size_t dyn_max = 0;
  if (m1_configure(prop.sharedMemPerBlockOptin, &dyn_max) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_OK;
  }
  l->smem_optin = dyn_max;
  {
    // low batch: the same descriptor (256-row boxes); v and x in fragment order per 512-column chunk,
    // then x at the salient columns; partial rows and counters of split 256-row tiles
    size_t mb_dyn = 0;
    const int mb_tiles = (l->N + kMbTileRows - 1) / kMbTileRows;
    // chunks, then (with salient columns) the prep kernel's residual per tile and x at the salient
    // columns for the helper warps
    const size_t ws = (size_t)l->n_chunks * kMbChunkWsBytes +
                      (l->n_salient > 0 ? (size_t)mb_tiles * kMbResFloatsPerTile * sizeof(float) +
                                              (size_t)16 * round_up(l->n_salient, 16) * 2
                                        : 0);
    const size_t ctr = (size_t)mb_tiles * kMbConsumerWarps * sizeof(unsigned);
    l->mb_ok = mb_configure(prop.sharedMemPerBlockOptin, &mb_dyn) == cudaSuccess &&
               mb_prep_configure(prop.sharedMemPerBlockOptin) == cudaSuccess;
    l->prep_smem_optin = prop.sharedMemPerBlockOptin;
    if (!l->mb_ok) cudaGetLastError();
    l->mb_smem_optin = mb_dyn;
    if (l->mb_ok) {
      if (cudaMalloc(&l->mb_ws, ws) != cudaSuccess ||
          cudaMalloc(&l->mb_part, (size_t)l->sm_count * kMbPartFloatsPerCta * sizeof(float)) != cudaSuccess ||
          cudaMalloc(&l->mb_counters, ctr) != cudaSuccess)
        return QTEA_ERR_ALLOC;
      if (cudaMemset(l->mb_counters, 0, ctr) != cudaSuccess) return QTEA_ERR_CUDA;
      // partial rows of split tiles: zero reads as "not written yet"; completed calls leave it zero
      if (cudaMemset(l->mb_part, 0, (size_t)l->sm_count * kMbPartFloatsPerCta * sizeof(float)) != cudaSuccess)
        return QTEA_ERR_CUDA;
      if (cudaMalloc(&l->mb_gbar, sizeof(unsigned long long)) != cudaSuccess) return QTEA_ERR_ALLOC;
      if (cudaMemset(l->mb_gbar, 0, sizeof(unsigned long long)) != cudaSuccess) return QTEA_ERR_CUDA;
      l->mb_gbar_next = 0;
    }
  }
  if (cudaMalloc(&l->workspace, (size_t)l->sm_count * 2 * kTileRows * sizeof(float)) != cudaSuccess)
    return QTEA_ERR_ALLOC;
  // split-tile partial rows: zero reads as "not written yet", and every completed call leaves it zero
  if (cudaMemset(l->workspace, 0, (size_t)l->sm_count * 2 * kTileRows * sizeof(float)) != cudaSuccess)
    return QTEA_ERR_CUDA;
  if (cudaMalloc(&l->counters, (size_t)l->n_tiles * kConsumerWarps * sizeof(unsigned)) != cudaSuccess)
    return QTEA_ERR_ALLOC;
  if (cudaMemset(l->counters, 0, (size_t)l->n_tiles * kConsumerWarps * sizeof(unsigned)) != cudaSuccess)
    return QTEA_ERR_CUDA;
  l->m1_ok = true;
  return QTEA_OK;
}

// Resources of the table-lookup kernel for a base-3 layout: split-tile workspace and counters.
int plan_lut(qtea_layout* l, const cudaDeviceProp& prop) {
  l->lut_ok = false;
  if (l->N == 0 || l->K == 0) return QTEA_OK;
  if (lut_configure(prop.sharedMemPerBlockOptin) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_OK;
  }
  const size_t tiles = (size_t)(l->N + kLutTileRows - 1) / kLutTileRows;
  const size_t ctr = tiles * kLutWarps * sizeof(unsigned);
  if (cudaMalloc(&l->lut_ws, (size_t)prop.multiProcessorCount * 2 * kLutTileRows * sizeof(float)) != cudaSuccess ||
      cudaMalloc(&l->lut_counters, ctr) != cudaSuccess)
    return QTEA_ERR_ALLOC;
  if (cudaMemset(l->lut_counters, 0, ctr) != cudaSuccess) return QTEA_ERR_CUDA;
  l->lut_ok = true;
  return QTEA_OK;
}

// The table-lookup kernel takes this batch-1 problem: base-3 codes (alpha per row or per group of
// 128 columns, with or without beta), the fixed-point kernel not asked for, and a chunk's share of
// the salient entries within its staging. (Measured on the Llama3-8B
// layer in base-3 codes: 63 us per step by table, 97 us by the fixed-point kernel.)
bool lut_eligible(const qtea_layout* l, int M) {
  if (M != 1 || !l->lut_ok || l->format != QTEA_FMT_BASE3 || (l->options & QTEA_OPT_FIXED_POINT)) return false;
  const int n_blocks = l->K_pad / 128, n_chunks = (n_blocks + kLutBlocks - 1) / kLutBlocks;
  const int nb = (l->n_salient + 7) / 8;
  return ((nb + n_chunks - 1) / n_chunks) * 8 <= kLutMaxEntries;
}

// Scale groups for the table-lookup kernel: alpha (and beta) staged per 128-column block, each
// block reading its group's pair; a layout with one alpha per row and no beta needs none.
bool lut_grouped(const qtea_layout* l) { return l->group_size != l->K || (l->options & QTEA_OPT_BIAS); }

// Table-lookup problems: consecutive problems of one variant (with or without scale groups), up to
// kMaxProblems, share a launch.
int run_lut(const qtea_gemv_problem* qs, const int* idx, int n, cudaStream_t st) {
  int i = 0;
  while (i < n) {
    LutParams P;
    std::memset(&P, 0, sizeof(P));
    const bool grouped = lut_grouped(qs[idx[i]].packed_ternary);
    int k = 0, sm_count = 1;
    while (i + k < n && k < kMaxProblems && lut_grouped(qs[idx[i + k]].packed_ternary) == grouped) {
      const qtea_gemv_problem& q = qs[idx[i + k]];
      const qtea_layout* l = q.packed_ternary;
      LutProblem& a = P.prob[k];
      a.x = q.x;
      a.packed = l->packed;
      a.scales = q.row_scale;
      a.v = q.col_scale;
      a.sal = q.salient_idx;
      a.rvals = q.residual_vals;
      a.ridx = q.residual_idx;
      a.y = q.y;
      a.ws = l->lut_ws;
      a.counters = l->lut_counters;
      a.N = l->N;
      a.K = l->K;
      a.s = l->n_salient;
      a.row_bytes = l->row_bytes;
      a.n_blocks = l->K_pad / 128;
      a.n_tiles = (l->N + kLutTileRows - 1) / kLutTileRows;
      a.n_chunks = (a.n_blocks + kLutBlocks - 1) / kLutBlocks;
      a.fp8 = (l->options & QTEA_OPT_RESIDUAL_FP8) ? 1 : 0;
      a.aligned8 = (l->row_bytes % 8 == 0 && aligned(l->packed, 8)) ? 1 : 0;
      a.G = (l->K + l->group_size - 1) / l->group_size;
      a.bias = (l->options & QTEA_OPT_BIAS) ? 1 : 0;
      a.gdiv = l->group_size == l->K ? a.n_blocks : 1;
      a.unit_begin = P.total_units;
      P.total_units += (long long)a.n_tiles * a.n_chunks;
      sm_count = l->sm_count;  // every layout records the device's SM count (its workspace's CTA slots)
      ++k;
    }
    P.n_problems = k;
    int grid = (int)(P.total_units < sm_count ? P.total_units : sm_count);
    if (grid > kMaxGrid) grid = kMaxGrid;
    for (int b = 0; b <= grid; ++b) P.cta_u0[b] = (int)unit_begin_of(b, P.total_units, grid);
    if (launch_lut(P, grouped, grid, st) != cudaSuccess) return QTEA_ERR_CUDA;
    i += k;
  }
  return QTEA_OK;
}

// Host-side checks of one problem; returns QTEA_OK or the status to report.
int check_problem(const qtea_gemv_problem& q, int M) {
  const qtea_layout* l = q.packed_ternary;
  if (!l) return QTEA_ERR_INVALID_ARG;
  if (M < 1 || M > QTEA_MAX_M) return QTEA_ERR_INVALID_ARG;
  if (l->N == 0) return QTEA_OK;
  if (!q.y || !aligned(q.y, 4)) return QTEA_ERR_INVALID_ARG;
  if (l->K == 0) return QTEA_OK;
  if (!q.x || !q.row_scale || !q.col_scale) return QTEA_ERR_INVALID_ARG;
  if (!aligned(q.x, 2) || !aligned(q.row_scale, 2) || !aligned(q.col_scale, 2)) return QTEA_ERR_INVALID_ARG;
  const size_t rv_align = (l->options & QTEA_OPT_RESIDUAL_FP8) ? 1 : 2;
  if (l->n_salient > 0 && (!q.salient_idx || !q.residual_vals || !q.residual_idx || !aligned(q.salient_idx, 4) ||
                           !aligned(q.residual_vals, rv_align)))
    return QTEA_ERR_INVALID_ARG;
  return QTEA_OK;
}

// The batch-1 kernel serves 2-bit layouts with fp16 residual values: one alpha per row, or alpha
// (and beta) per group of 128 columns or per row (its grouped variant).
bool m1_capable(const qtea_layout* l) {
  return l->format == QTEA_FMT_2BIT && !(l->options & QTEA_OPT_RESIDUAL_FP8) &&
         (l->group_size == l->K || l->group_size == 128);
}

// The paper's own storage: base-3 codes, groups of 128 columns, beta or FP8 residual values.
bool is_paper(const qtea_layout* l) {
  return l->format != QTEA_FMT_2BIT || l->group_size != l->K ||
         (l->options & (QTEA_OPT_BIAS | QTEA_OPT_RESIDUAL_FP8)) != 0;
}

PaperParams paper_params(const qtea_gemv_problem& q, int M) {
  const qtea_layout* l = q.packed_ternary;
  PaperParams p;
  p.x = q.x;
  p.packed = l->packed;
  p.scales = q.row_scale;
  p.v = q.col_scale;
  p.sal = q.salient_idx;
  p.rvals = q.residual_vals;
  p.ridx = q.residual_idx;
  p.y = q.y;
  p.M = M;
  p.N = l->N;
  p.K = l->K;
  p.s = l->n_salient;
  p.group_size = l->group_size > 0 ? l->group_size : 1;
  p.G = (l->K + p.group_size - 1) / p.group_size;
  p.row_bytes = l->row_bytes;
  p.format = l->format;
  p.bias = (l->options & QTEA_OPT_BIAS) ? 1 : 0;
  p.residual_fp8 = (l->options & QTEA_OPT_RESIDUAL_FP8) ? 1 : 0;
  p.staged_ok = l->paper_staged_ok ? 1 : 0;
  p.sm_count = l->sm_count > 0 ? l->sm_count : 1;
  p.smem_optin = l->smem_optin;
  p.smem_per_sm = l->smem_per_sm;
  return p;
}

int launch_paper_problem(const qtea_gemv_problem& q, int M, cudaStream_t st) {
  return launch_paper(paper_params(q, M), st) == cudaSuccess ? QTEA_OK : QTEA_ERR_CUDA;
}

// Base-3 problems with staged activations: up to eight per launch.
int run_b3(const qtea_gemv_problem* qs, const int* idx, int n, int M, cudaStream_t st) {
  for (int i = 0; i < n; i += 8) {
    B3Group g;
    g.n = n - i < 8 ? n - i : 8;
    g.work[0] = 0;
    for (int k = 0; k < g.n; ++k) {
      g.prob[k] = paper_params(qs[idx[i + k]], M);
      g.work[k + 1] = g.work[k] + (long long)g.prob[k].N * ((g.prob[k].K + 127) / 128);
    }
    if (launch_b3(g, st) != cudaSuccess) return QTEA_ERR_CUDA;
  }
  return QTEA_OK;
}

int launch_generic_problem(const qtea_gemv_problem& q, int M, cudaStream_t st) {
  const qtea_layout* l = q.packed_ternary;
  GenericParams p;
  p.x = q.x;
  p.packed = l->packed;
  p.alpha = q.row_scale;
  p.v = q.col_scale;
  p.sal = q.salient_idx;
  p.rvals = q.residual_vals;
  p.ridx = q.residual_idx;
  p.y = q.y;
  p.M = M;
  p.N = l->N;
  p.K = l->K;
  p.K_pad = l->K_pad;
  p.s = l->n_salient;
  return launch_generic(p, st) == cudaSuccess ? QTEA_OK : QTEA_ERR_CUDA;
}

// Low-batch (2 <= M <= 16) problems on the tensor-core kernel, up to kMaxProblems per launch: one
// prep launch writes v and x of every problem in fragment order into the layouts' workspaces, one
// main launch streams the codes of all of them.
struct MbGroup {
  MbGroupParams gp;
  MbPrepGroup pg;
  TensorMaps maps;
  int grid = 0;
  size_t smem = 0;
  size_t prep_smem_optin = 0;
  size_t smem_optin = 0;  // the main kernel's dynamic shared memory limit
  TensorMaps ab_maps;     // scale groups: alpha (and beta) per row and 128-column group
  bool grp = false;       // the group's problems have scale groups (one kernel variant per launch)
};

void mb_group_reset(MbGroup& g, int M, size_t prep_smem_optin, size_t smem_optin) {
  std::memset(&g.gp, 0, sizeof(g.gp));
  std::memset(&g.pg, 0, sizeof(g.pg));
  std::memset(&g.maps, 0, sizeof(g.maps));
  std::memset(&g.ab_maps, 0, sizeof(g.ab_maps));
  g.grp = false;
  g.gp.M = M;
  g.pg.M = M;
  g.pg.mt = mb_mt(M);
  g.gp.split = g.pg.split = mb_split(M) ? 1 : 0;
  g.grid = 0;
  g.smem = 0;
  g.prep_smem_optin = prep_smem_optin;
  g.smem_optin = smem_optin;
}

// Scale groups of the low-batch kernel: row_scale as [N][G] alpha or [N][2G] (alpha, beta) fp16
// for TMA boxes of 8 values x 256 rows; false if its address or row stride does not allow them.
bool encode_ab_map(const qtea_layout* l, const uint16_t* row_scale, CUtensorMap* out) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = get_encode_tiled();
  if (!encode || !aligned(row_scale, 16)) return false;
  const int G = (l->K + 127) / 128;
  const int cols = G * ((l->options & QTEA_OPT_BIAS) ? 2 : 1);
  if ((cols * 2) % 16 != 0) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)l->N};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {8, (cuuint32_t)kMbTileRows};
  cuuint32_t estr[2] = {1, 1};
  return encode(out, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<uint16_t*>(row_scale), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool mb_group_add(MbGroup& g, const qtea_gemv_problem& q) {
  if (g.gp.n_problems == kMaxProblems) return false;
  const qtea_layout* l = q.packed_ternary;
  const int k = g.gp.n_problems;
  const bool grp = l->group_size != l->K;
  if (k > 0 && grp != g.grp) return false;
  if (grp && !encode_ab_map(l, q.row_scale, &g.ab_maps.m[k])) return false;
  g.grp = grp;
  const int n_tiles = (l->N + kMbTileRows - 1) / kMbTileRows;
  const int s = l->n_salient, s16 = round_up(s, 16);
  const int mt = mb_mt(g.gp.M);
  uint8_t* res_base = l->mb_ws + (size_t)l->n_chunks * kMbChunkWsBytes;
  float* yres = s > 0 ? reinterpret_cast<float*>(res_base) : nullptr;
  uint16_t* xs = s > 0 ? reinterpret_cast<uint16_t*>(res_base + (size_t)n_tiles * kMbResFloatsPerTile * sizeof(float))
                       : nullptr;
  // residual by the main kernel's helpers when the caller's arrays allow bulk copies and a pass over a
  // half or quarter of a tile's row groups fits beside two code stages; else by the prep kernel
  const bool fp8 = (l->options & QTEA_OPT_RESIDUAL_FP8) != 0;
  int mode = s > 0 ? kMbResPrep : kMbResNone, passes = 0;
  if (s > 0 && aligned(q.residual_vals, 16) && aligned(q.residual_idx, 16)) {
    for (int p = 1; p <= 4 && !passes; p *= 2)
      if (mb_smem_layout(kMinStagesMb, mt, grp, (int)mb_res_stage_bytes(s, p, fp8)).total <= g.smem_optin) passes = p;
    if (passes) mode = kMbResHelpers;
  }
  if (fp8 && mode == kMbResPrep) return false;  // FP8 values only through the helpers
  MbPrepProblem& pp = g.pg.prob[k];
  pp.x = q.x;
  pp.v = q.col_scale;
  pp.sal = q.salient_idx;
  pp.rvals = q.residual_vals;
  pp.ridx = q.residual_idx;
  pp.ws = l->mb_ws;
  pp.yres = yres;
  pp.xs = xs;
  pp.N = l->N;
  pp.K = l->K;
  pp.s = s;
  pp.s16 = s16;
  pp.n_chunks = l->n_chunks;
  pp.n_tiles = n_tiles;
  pp.res_mode = mode;
  pp.native = mode == kMbResPrep && aligned(q.residual_vals, 16) && aligned(q.residual_idx, 16) &&
              mb_prep_smem_bytes(s, true) <= g.prep_smem_optin;
  pp.block_begin = g.pg.n_blocks;
  const size_t need = mb_prep_smem_bytes(mode == kMbResPrep ? s : 0, pp.native != 0);
  if (need > g.pg.smem) g.pg.smem = need;
  MbProblemArgs& a = g.gp.prob[k];
  a.alpha = q.row_scale;
  a.ws = l->mb_ws;
  a.yres = yres;
  a.rvals = q.residual_vals;
  a.ridx = q.residual_idx;
  a.xs = xs;
  a.y = q.y;
  a.part = l->mb_part;
  a.counters = l->mb_counters;
  a.N = l->N;
  a.n_tiles = n_tiles;
  a.n_chunks = l->n_chunks;
  a.s = s;
  a.s16 = s16;
  a.res_mode = mode;
  a.res_passes = passes;
  a.bias = (l->options & QTEA_OPT_BIAS) ? 1 : 0;
  a.fp8 = fp8 ? 1 : 0;
  a.unit_begin = g.gp.total_units;
  if (mode == kMbResHelpers) {
    const int rsb = (int)mb_res_stage_bytes(s, passes, fp8);
    if (rsb > g.gp.res_stage_bytes) g.gp.res_stage_bytes = rsb;
  }
  std::memcpy(&g.maps.m[k], &l->tmap, sizeof(CUtensorMap));
  if (k == 0) g.gp.status = l->status;
  g.gp.total_units += (long long)a.n_tiles * a.n_chunks;
  g.pg.n_blocks += l->n_chunks + (mode == kMbResPrep ? n_tiles : mode == kMbResHelpers ? (s16 + 255) / 256 : 0);
  g.gp.n_problems += 1;
  g.pg.n_problems += 1;
  return true;
}

// Grid, ring depth and shared memory of the group; false if the ring does not fit.
bool mb_group_plan(MbGroup& g, int sm_count, size_t smem_optin) {
  if (g.gp.n_problems == 0) return false;
  if (g.gp.total_units >= (1ll << 30)) return false;
  g.grid = (int)(g.gp.total_units < sm_count ? g.gp.total_units : sm_count);
  if (g.grid > kMaxGrid) g.grid = kMaxGrid;
  for (int b = 0; b <= g.grid; ++b) g.gp.cta_u0[b] = (int)unit_begin_of(b, g.gp.total_units, g.grid);
  // no residual left to the prep kernel: its other work moves into the main kernel (one launch)
  g.gp.fused = 1;
  for (int k = 0; k < g.gp.n_problems; ++k)
    if (g.gp.prob[k].res_mode == kMbResPrep) g.gp.fused = 0;
  if (g.gp.fused) {
    g.gp.prep = g.pg;
    const int scratch = kMbPrepScratch;  // the chunk build's
    if (g.gp.res_stage_bytes < scratch) g.gp.res_stage_bytes = scratch;
  }
  for (int S = kMaxStagesMb; S >= kMinStagesMb; --S) {
    const size_t bytes = mb_smem_bytes(S, g.gp.M, g.grp, g.gp.res_stage_bytes);
    if (bytes <= smem_optin) {
      g.gp.n_stages = S;
      g.smem = bytes;
      return true;
    }
  }
  return false;
}

int mb_group_launch(MbGroup& g, const qtea_layout* l0, cudaStream_t st) {
  if (g.gp.fused) {
    // the barrier counter only grows: this launch's CTAs wait for it to reach the value after them
    g.gp.gbar = l0->mb_gbar;
    l0->mb_gbar_next += (unsigned long long)g.grid;
    g.gp.gbar_target = l0->mb_gbar_next;
  } else if (launch_mb_prep(g.pg, st) != cudaSuccess) {
    return QTEA_ERR_CUDA;
  }
  return launch_mb(g.maps, g.ab_maps, g.gp, g.grp, g.grid, g.smem, st) == cudaSuccess ? QTEA_OK : QTEA_ERR_CUDA;
}

// The low-batch kernel serves the library's own layouts at 2 <= M <= 16 and, at any M, layouts in
// the paper's storage with 2-bit codes, fp16 or FP8 residual values, and one alpha per row or alpha
// (and beta) per 128-column group.
bool mb_capable(const qtea_layout* l, int M) {
  if (!l->mb_ok || !l->m1_ok || M < 1 || M > 16) return false;
  if (!is_paper(l)) return M >= 2;
  if (l->format != QTEA_FMT_2BIT) return false;
  return l->group_size == 128 || !(l->options & QTEA_OPT_BIAS);
}

// Low-batch dispatch: as many consecutive problems per launch as fit (one kernel variant per
// launch); a problem the kernel cannot take goes to the paper-storage or the generic kernel.
int run_mb(const qtea_gemv_problem* qs, const int* idx, int n, int M, cudaStream_t st) {
  int i = 0;
  while (i < n) {
    const qtea_layout* l0 = qs[idx[i]].packed_ternary;
    MbGroup g;
    mb_group_reset(g, M, l0->prep_smem_optin, l0->mb_smem_optin);
    int taken = 0;
    while (i + taken < n) {
      const qtea_layout* li = qs[idx[i + taken]].packed_ternary;
      if (li->sm_count != l0->sm_count) break;  // partial-row slots are sized by the SM count
      MbGroup trial = g;
      if (!mb_group_add(trial, qs[idx[i + taken]])) break;
      if (!mb_group_plan(trial, l0->sm_count, l0->mb_smem_optin)) break;
      g = trial;
      ++taken;
    }
    if (taken == 0) {
      int rc = is_paper(l0) ? launch_paper_problem(qs[idx[i]], M, st) : launch_generic_problem(qs[idx[i]], M, st);
      if (rc) return rc;
      ++i;
      continue;
    }
    int rc = mb_group_launch(g, l0, st);
    if (rc) return rc;
    i += taken;
  }
  return QTEA_OK;
}

// Batch-1 kernel over a group of problems whose layouts all have m1 resources.
struct M1Group {
  GroupParams gp;
  TensorMaps maps;
  int grid = 0;
  size_t smem = 0;
};

void group_reset(M1Group& g) {
  std::memset(&g.gp, 0, sizeof(g.gp));
  g.gp.n_problems = 0;
  g.gp.total_units = 0;
}

// The batch-1 kernels' record of problem q (the split-tile fields point at the layout's resources).
ProblemArgs problem_args(const qtea_gemv_problem& q) {
  const qtea_layout* l = q.packed_ternary;
  ProblemArgs a;
  std::memset(&a, 0, sizeof(a));
  a.x = q.x;
  a.alpha = q.row_scale;
  a.v = q.col_scale;
  a.sal = q.salient_idx;
  a.rvals = q.residual_vals;
  a.ridx = q.residual_idx;
  a.y = q.y;
  a.ws = l->workspace;
  a.counters = l->counters;
  a.N = l->N;
  a.K = l->K;
  a.s = l->n_salient;
  a.n_tiles = l->n_tiles;
  a.n_chunks = l->n_chunks;
  a.act_bits = (l->act_bits == 16 && l->K >= kMinK16) ? 16 : 24;
  const bool bias = (l->options & QTEA_OPT_BIAS) != 0, groups = l->group_size != l->K || bias;
  a.G = (l->K + l->group_size - 1) / l->group_size;
  a.gdiv = l->group_size == l->K ? l->n_chunks * 4 : 1;  // 128-column groups per scale group
  const bool vec = groups && a.gdiv == 1 && a.G % 4 == 0 && aligned(q.row_scale, bias ? 16 : 8);
  a.gflags = (groups ? kScaleGroups : 0) | (bias ? kScaleBias : 0) | (vec ? kScaleVec : 0);
  a.vec_xv = aligned(q.x, 16) && aligned(q.col_scale, 16);
  a.vec_res = (l->n_salient % kResBlock == 0) && aligned(q.residual_vals, 16) && aligned(q.residual_idx, 2);
  return a;
}

// Add problem q; false if the group is full.
bool group_add(M1Group& g, const qtea_gemv_problem& q) {
  if (g.gp.n_problems == kMaxProblems) return false;
  const qtea_layout* l = q.packed_ternary;
  ProblemArgs& a = g.gp.prob[g.gp.n_problems];
  a = problem_args(q);
  a.unit_begin = g.gp.total_units;
  if (a.gflags & kScaleGroups) g.gp.n_grp += 1;
  std::memcpy(&g.maps.m[g.gp.n_problems], &l->tmap, sizeof(CUtensorMap));
  if (g.gp.n_problems == 0) g.gp.status = l->status;
  g.gp.total_units += (long long)l->n_tiles * l->n_chunks;
  g.gp.n_problems += 1;
  return true;
}

// Grid, ring depth and shared memory of the group; false if the ring does not fit.
bool group_plan(M1Group& g, int sm_count, size_t smem_optin) {
  if (g.gp.n_problems == 0) return false;
  if (g.gp.total_units >= (1ll << 30)) return false;
  g.grid = (int)(g.gp.total_units < sm_count ? g.gp.total_units : sm_count);
  if (g.grid > kMaxGrid) g.grid = kMaxGrid;
  for (int b = 0; b <= g.grid; ++b) g.gp.cta_u0[b] = (int)unit_begin_of(b, g.gp.total_units, g.grid);
  for (int stages = kMaxStages; stages >= kMinStages; --stages) {
    if (m1_smem_bytes(stages) <= smem_optin) {
      g.gp.n_stages = stages;
      g.smem = m1_smem_bytes(stages);
      return true;
    }
  }
  return false;
}

int group_launch(M1Group& g, cudaStream_t st) {
  return launch_m1(g.maps, g.gp, g.grid, g.smem, st) == cudaSuccess ? QTEA_OK : QTEA_ERR_CUDA;
}

// Batch-1 dispatch: pack as many consecutive problems as fit into each launch. caller_codes: the
// packed codes belong to the caller, so the kernel reads them only after the grid dependency wait.
int run_m1(const qtea_gemv_problem* qs, const int* idx, int n, cudaStream_t st, bool caller_codes = false) {
  int i = 0;
  while (i < n) {
    const qtea_layout* l0 = qs[idx[i]].packed_ternary;
    M1Group g;
    group_reset(g);
    g.gp.codes_after_wait = caller_codes ? 1 : 0;
    int taken = 0;
    while (i + taken < n) {
      M1Group trial = g;
      if (!group_add(trial, qs[idx[i + taken]])) break;
      if (!group_plan(trial, l0->sm_count, l0->smem_optin)) break;
      g = trial;
      ++taken;
    }
    if (taken == 0) {
      // the ring does not fit this device's shared memory: the generic kernel serves the problem
      int rc = launch_generic_problem(qs[idx[i]], 1, st);
      if (rc) return rc;
      ++i;
      continue;
    }
    int rc = group_launch(g, st);
    if (rc) return rc;
    i += taken;
  }
  return QTEA_OK;
}

// ---------------------------------------------------------------- row-resident batch-1 kernel
// Layouts it may serve: 2-bit codes, one alpha per row, fp16 residual values, at most
// kRowsMaxChunks 512-column chunks and kRowsMaxSalientWide salient columns, not pinned to the
// stream-K kernel. Beyond one chunk per warp or kRowsMaxSalient salient columns a launch is wide.
bool rows_shape_ok(int n_chunks, int s) { return n_chunks <= kRowsMaxChunks && s <= kRowsMaxSalientWide; }
bool rows_shape_wide(int n_chunks, int s) { return n_chunks > kRowsWarps || s > kRowsMaxSalient; }
bool rows_capable(const qtea_layout* l) {
  return l->rows_ok && l->m1_ok && l->format == QTEA_FMT_2BIT && l->group_size == l->K &&
         (l->options & (QTEA_OPT_BIAS | QTEA_OPT_RESIDUAL_FP8 | QTEA_OPT_STREAM_K)) == 0 &&
         rows_shape_ok(l->n_chunks, l->n_salient);
}

struct RowsLaunch {
  RowsParams rp;
  TensorMaps maps;
  int grid = 0;
  size_t smem = 0;
};

// CTAs per problem for a grid of at most `ctas`: in proportion to its codes (at least one), then
// one at a time to the problem with the most codes per CTA. Returns the rows of the largest CTA.
long long rows_split(const long long* blocks, const int* chunks, int n, int ctas, int* cnt) {
  long long total = 0;
  for (int i = 0; i < n; ++i) total += blocks[i] * chunks[i];
  int used = 0;
  for (int i = 0; i < n; ++i) {
    long long c = (long long)ctas * blocks[i] * chunks[i] / total;
    if (c < 1) c = 1;
    if (c > blocks[i]) c = blocks[i];
    cnt[i] = (int)c;
    used += cnt[i];
  }
  auto cost = [&](int i) { return (blocks[i] + cnt[i] - 1) / cnt[i] * chunks[i]; };
  while (used > ctas) {  // the one-CTA minimums overshot: take from the cheapest per CTA
    int best = -1;
    for (int i = 0; i < n; ++i)
      if (cnt[i] > 1 && (best < 0 || cost(i) < cost(best))) best = i;
    if (best < 0) return -1;
    --cnt[best];
    --used;
  }
  while (used < ctas) {
    int best = -1;
    for (int i = 0; i < n; ++i)
      if (cnt[i] < blocks[i] && (best < 0 || cost(i) > cost(best))) best = i;
    if (best < 0) break;
    ++cnt[best];
    ++used;
  }
  long long rows = 0;
  for (int i = 0; i < n; ++i) {
    const long long r = (blocks[i] + cnt[i] - 1) / cnt[i] * kRowsBoxRows;
    rows = r > rows ? r : rows;
  }
  return rows;
}

// The shape of a row-resident launch for n problems (rows N[i], chunks nch[i], salient columns s[i])
// on a device of sm SMs with smem_optin bytes of shared memory per CTA: one CTA per SM where that
// leaves every CTA kRowsMaxRows rows or fewer (one per lane), else two CTAs per SM (not for a wide
// launch). False if the problems do not fit: a shape beyond the kernel's limits, more problems than
// CTAs, more than kRowsMaxRows rows in a CTA, or shared memory beyond the device's limit.
struct RowsShapePlan {
  int cnt[kMaxProblems];  // CTAs of each problem
  int grid, rows_cap, nch_max, kparts;
  bool wide;
  size_t smem;
};
bool rows_plan_shapes(const long long* N, const int* nch, const int* s, int n, int sm, size_t smem_optin,
                      RowsShapePlan& P) {
  if (n < 1 || n > kMaxProblems || sm < 1 || n > sm || 2 * sm > kMaxGrid) return false;
  long long blocks[kMaxProblems];
  P.nch_max = 0;
  P.wide = false;
  for (int i = 0; i < n; ++i) {
    if (N[i] < 1 || nch[i] < 1 || s[i] < 0 || !rows_shape_ok(nch[i], s[i])) return false;
    blocks[i] = (N[i] + kRowsBoxRows - 1) / kRowsBoxRows;
    P.nch_max = nch[i] > P.nch_max ? nch[i] : P.nch_max;
    P.wide = P.wide || rows_shape_wide(nch[i], s[i]);
  }
  long long rows_cap = rows_split(blocks, nch, n, sm, P.cnt);
  if (rows_cap > kRowsMaxRows && !P.wide) {
    int cnt2[kMaxProblems];
    const long long r2 = rows_split(blocks, nch, n, 2 * sm, cnt2);
    if (r2 > 0 && r2 <= kRowsMaxRows) {
      rows_cap = r2;
      for (int i = 0; i < n; ++i) P.cnt[i] = cnt2[i];
    }
  }
  if (rows_cap < 1 || rows_cap > kRowsMaxRows) return false;
  const RowsSmem so = rows_smem_layout((int)rows_cap, P.nch_max);
  if (so.total > smem_optin) return false;
  // lanes per row (4 for up to 8 rows, 2 for 16, 1 for more): one value for every CTA, or 0
  int kp = -1;
  P.grid = 0;
  for (int i = 0; i < n; ++i) {
    P.grid += P.cnt[i];
    for (int j = 0; j < P.cnt[i] && kp != 0; ++j) {
      const long long r0 = blocks[i] * j / P.cnt[i] * kRowsBoxRows, r1 = blocks[i] * (j + 1) / P.cnt[i] * kRowsBoxRows;
      const long long R = (r1 < N[i] ? r1 : N[i]) - r0;
      const int k = R <= 8 ? 4 : R <= 16 ? 2 : 1;
      if (kp < 0) kp = k;
      else if (kp != k) kp = 0;
    }
  }
  P.kparts = kp < 0 ? 0 : kp;
  P.rows_cap = (int)rows_cap;
  P.smem = so.total;
  return true;
}

// One row-resident launch for problems idx[0 .. n), planned by rows_plan_shapes; false if a layout
// cannot take the kernel or the problems do not fit one launch.
bool rows_plan(const qtea_gemv_problem* qs, const int* idx, int n, RowsLaunch& L) {
  if (n < 1 || n > kMaxProblems) return false;
  const qtea_layout* l0 = qs[idx[0]].packed_ternary;
  long long N[kMaxProblems];
  int nch[kMaxProblems], sal[kMaxProblems];
  for (int i = 0; i < n; ++i) {
    const qtea_layout* l = qs[idx[i]].packed_ternary;
    if (!rows_capable(l) || l->sm_count != l0->sm_count || l->device != l0->device) return false;
    N[i] = l->N;
    nch[i] = l->n_chunks;
    sal[i] = l->n_salient;
  }
  RowsShapePlan P;
  if (!rows_plan_shapes(N, nch, sal, n, l0->sm_count, l0->rows_smem_optin, P)) return false;
  std::memset(&L.rp, 0, sizeof(L.rp));
  int b = 0;
  for (int i = 0; i < n; ++i) {
    const qtea_gemv_problem& q = qs[idx[i]];
    L.rp.prob[i] = problem_args(q);
    L.rp.cta_begin[i] = b;
    b += P.cnt[i];
    std::memcpy(&L.maps.m[i], &q.packed_ternary->tmap8, sizeof(CUtensorMap));
  }
  L.rp.cta_begin[n] = b;
  L.rp.kparts = P.kparts;
  L.rp.wide = P.wide ? 1 : 0;
  L.rp.rows_cap = P.rows_cap;
  L.rp.n_chunks_max = P.nch_max;
  L.rp.n_problems = n;
  L.rp.status = l0->status;
  L.grid = b;
  L.smem = P.smem;
  return true;
}

// Batch-1 dispatch of problems idx[0 .. n): one row-resident launch when all of them fit it, else
// the stream-K kernel.
int run_batch1(const qtea_gemv_problem* qs, const int* idx, int n, cudaStream_t st) {
  RowsLaunch L;
  if (rows_plan(qs, idx, n, L))
    return launch_rows(L.maps, L.rp, L.grid, L.smem, st) == cudaSuccess ? QTEA_OK : QTEA_ERR_CUDA;
  return run_m1(qs, idx, n, st);
}

// ---------------------------------------------------------------- allocation-free batch-1 entry
// qtea_gemv_m1_static serves callers that may not allocate device memory. Its split-tile scratch is
// this fixed array in static device memory (one copy per device), laid out as
//   [0, kStaticWsBytes)             partial sums   [kStaticGrid][2][kTileRows], zero between calls
//   [kStaticWsBytes, +kStaticCtrBytes)  counters   [kStaticTiles][kConsumerWarps] unsigned, zero
//   then the status word (int)
// The scratch starts at zero because static device memory is zero-initialised when the module is
// loaded, and every completed call leaves it at zero (the CTA that sums a split tile zeroes the
// partial rows it read).
constexpr int kStaticGrid = 160;                 // CTAs a call may use (>= the 152 SMs of a GB300)
constexpr int kStaticTiles = 256;                // 512-row tiles: N <= 131072
constexpr size_t kStaticWsBytes = (size_t)kStaticGrid * 2 * kTileRows * sizeof(float);    // 655,360
constexpr size_t kStaticCtrBytes = (size_t)kStaticTiles * kConsumerWarps * sizeof(unsigned);  // 8,192
constexpr size_t kStaticScratchBytes = kStaticWsBytes + kStaticCtrBytes + 256;              // 663,808
constexpr int kStaticMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Per-device set-up, done once with that device current: the scratch address, the SM count and
// the batch-1 kernel's shared-memory limit.
struct StaticDevice {
  bool ready = false;
  bool m1_ok = false;
  unsigned char* scratch = nullptr;
  int sm_count = 0;
  size_t smem_optin = 0;
};
StaticDevice g_static_dev[kStaticMaxDevices];
std::mutex g_static_mu;

int static_setup(int dev, StaticDevice* out) {
  std::lock_guard<std::mutex> lock(g_static_mu);
  StaticDevice& d = g_static_dev[dev];
  if (!d.ready) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return QTEA_ERR_CUDA;
    }
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) {
      cudaGetLastError();
      return QTEA_ERR_CUDA;
    }
    size_t dyn_max = 0;
    d.m1_ok = get_encode_tiled() != nullptr && m1_configure(prop.sharedMemPerBlockOptin, &dyn_max) == cudaSuccess;
    if (!d.m1_ok) cudaGetLastError();
    d.scratch = static_cast<unsigned char*>(p);
    d.sm_count = prop.multiProcessorCount < kStaticGrid ? prop.multiProcessorCount : kStaticGrid;
    d.smem_optin = dyn_max;
    d.ready = true;
  }
  *out = d;
  return QTEA_OK;
}

}  // namespace

extern "C" {

const char* qtea_status_string(int status) {
  switch (status) {
    case QTEA_OK: return "success";
    case QTEA_ERR_INVALID_ARG: return "invalid argument";
    case QTEA_ERR_BAD_CODES: return "ternary code outside {-1, 0, +1}";
    case QTEA_ERR_UNSUPPORTED: return "unsupported request";
    case QTEA_ERR_CUDA: return "CUDA runtime error";
    case QTEA_ERR_ALLOC: return "device allocation failed";
    case QTEA_ERR_TIMEOUT: return "bounded wait in a kernel timed out";
    case QTEA_ERR_SCRATCH_LIMIT: return "problem larger than the static scratch of qtea_gemv_m1_static";
    case QTEA_ERR_STATE: return "static scratch of qtea_gemv_m1_static not in its start state (overlapping calls?)";
    default: return "unknown status";
  }
}

int qtea_pack_layout(const int8_t* ternary_codes, int N, int K, int group_size, int n_salient, int format,
                     qtea_stream_t stream, qtea_layout** out) {
  if (!out) return QTEA_ERR_INVALID_ARG;
  *out = nullptr;
  if (N < 0 || K < 0 || n_salient < 0 || n_salient > K) return QTEA_ERR_INVALID_ARG;
  if ((long long)N * K > 0 && !ternary_codes) return QTEA_ERR_INVALID_ARG;
  if (n_salient > 0 && N % 4 != 0) return QTEA_ERR_INVALID_ARG;
  if (format != QTEA_FMT_2BIT && format != QTEA_FMT_BASE3) return QTEA_ERR_INVALID_ARG;
  if (group_size != K && group_size != 128) return QTEA_ERR_UNSUPPORTED;
  if ((long long)K + 63 > 0x7fffffffLL) return QTEA_ERR_INVALID_ARG;

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return QTEA_ERR_CUDA; }
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) { cudaGetLastError(); return QTEA_ERR_CUDA; }

  qtea_layout* l = new (std::nothrow) qtea_layout;
  if (!l) return QTEA_ERR_ALLOC;
  std::memset(l, 0, sizeof(*l));
  l->N = N;
  l->K = K;
  l->K_pad = format == QTEA_FMT_BASE3 ? round_up(K, 128) : round_up(K, 64);
  l->group_size = group_size;
  l->n_salient = n_salient;
  l->format = format;
  l->options = 0;
  l->row_bytes = format == QTEA_FMT_BASE3 ? l->K_pad / 128 * 26 : l->K_pad / 4;
  l->device = dev;
  l->act_bits = 16;
  l->sm_count = prop.multiProcessorCount;
  l->smem_optin = prop.sharedMemPerBlockOptin;
  l->smem_per_sm = prop.sharedMemPerMultiprocessor;
  l->paper_staged_ok = paper_configure(prop.sharedMemPerBlockOptin) == cudaSuccess;
  if (!l->paper_staged_ok) cudaGetLastError();
  l->packed_bytes = (size_t)N * (size_t)l->row_bytes;
  if (cudaMalloc(&l->packed, l->packed_bytes > 0 ? l->packed_bytes : 16) != cudaSuccess ||
      cudaMalloc(&l->status, 2 * sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    release(l);
    return QTEA_ERR_ALLOC;
  }
  int rc = QTEA_OK;
  int host_flags[2] = {0, 0};
  if (cudaMemsetAsync(l->status, 0, 2 * sizeof(int), st) != cudaSuccess ||
      (format == QTEA_FMT_BASE3
           ? launch_pack_base3(ternary_codes, N, K, l->packed, l->status + 1, st)
           : launch_pack(ternary_codes, N, K, l->K_pad, reinterpret_cast<uint32_t*>(l->packed), l->status + 1, st)) !=
          cudaSuccess ||
      cudaMemcpyAsync(host_flags, l->status, sizeof(host_flags), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess) {
    rc = QTEA_ERR_CUDA;
  } else if (host_flags[1] != 0) {
    rc = QTEA_ERR_BAD_CODES;
  } else if (cudaMemsetAsync(l->status, 0, 2 * sizeof(int), st) != cudaSuccess) {
    rc = QTEA_ERR_CUDA;
  } else if (format == QTEA_FMT_2BIT) {
    rc = plan_m1(l, prop);  // the batch-1 and low-batch kernels' resources
  } else {
    rc = plan_lut(l, prop);  // the table-lookup kernel's resources
  }
  if (rc == QTEA_OK && cudaStreamSynchronize(st) != cudaSuccess) rc = QTEA_ERR_CUDA;
  if (rc != QTEA_OK) {
    cudaGetLastError();
    release(l);
    return rc;
  }
  *out = l;
  return QTEA_OK;
}

namespace {

// Which path serves problem q at batch M (before the batch-1 choice between the two launch forms).
enum Route { kRouteNone, kRouteZero, kRouteBatch1, kRouteLut, kRouteMb, kRouteB3, kRoutePaper, kRouteGeneric };

Route route(const qtea_gemv_problem& q, int M) {
  const qtea_layout* l = q.packed_ternary;
  if (l->N == 0) return kRouteNone;
  if (l->K == 0) return kRouteZero;
  if (M == 1 && l->m1_ok && m1_capable(l)) return kRouteBatch1;
  if (lut_eligible(l, M)) return kRouteLut;
  if (mb_capable(l, M)) return kRouteMb;
  if (is_paper(l)) return b3_eligible(paper_params(q, M)) ? kRouteB3 : kRoutePaper;
  return kRouteGeneric;
}

int check_call(const qtea_gemv_problem* problems, int n_problems, int M) {
  if (n_problems < 0 || (n_problems > 0 && !problems)) return QTEA_ERR_INVALID_ARG;
  if (M < 1 || M > QTEA_MAX_M) return QTEA_ERR_INVALID_ARG;
  for (int i = 0; i < n_problems; ++i) {
    int rc = check_problem(problems[i], M);
    if (rc) return rc;
    for (int j = 0; j < i; ++j)  // a layout's split-K workspace serves one problem per call
      if (problems[j].packed_ternary == problems[i].packed_ternary) return QTEA_ERR_INVALID_ARG;
  }
  return QTEA_OK;
}

}  // namespace

int qtea_gemv_grouped(const qtea_gemv_problem* problems, int n_problems, int M, qtea_stream_t stream) {
  int rc = check_call(problems, n_problems, M);
  if (rc) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int* m1_idx = n_problems > 0 ? static_cast<int*>(std::malloc(sizeof(int) * 2 * (size_t)n_problems)) : nullptr;
  if (n_problems > 0 && !m1_idx) return QTEA_ERR_ALLOC;
  int* mb_idx = m1_idx + n_problems;
  int b3_idx[8];
  int n_m1 = 0, n_mb = 0, n_b3 = 0, n_lut = 0;
  int lut_idx[kMaxProblems];
  for (int i = 0; i < n_problems && rc == QTEA_OK; ++i) {
    const qtea_gemv_problem& q = problems[i];
    switch (route(q, M)) {
      case kRouteNone:
        break;
      case kRouteZero:
        if (cudaMemsetAsync(q.y, 0, (size_t)M * q.packed_ternary->N * sizeof(float), st) != cudaSuccess)
          rc = QTEA_ERR_CUDA;
        break;
      case kRouteBatch1:
        m1_idx[n_m1++] = i;
        break;
      case kRouteLut:
        lut_idx[n_lut++] = i;
        if (n_lut == kMaxProblems) {
          rc = run_lut(problems, lut_idx, n_lut, st);
          n_lut = 0;
        }
        break;
      case kRouteMb:
        mb_idx[n_mb++] = i;
        break;
      case kRouteB3:
        b3_idx[n_b3++] = i;
        if (n_b3 == 8) {
          rc = run_b3(problems, b3_idx, n_b3, M, st);
          n_b3 = 0;
        }
        break;
      case kRoutePaper:
        rc = launch_paper_problem(q, M, st);
        break;
      case kRouteGeneric:
        rc = launch_generic_problem(q, M, st);
        break;
    }
  }
  if (rc == QTEA_OK && n_b3 > 0) rc = run_b3(problems, b3_idx, n_b3, M, st);
  if (rc == QTEA_OK && n_lut > 0) rc = run_lut(problems, lut_idx, n_lut, st);
  if (rc == QTEA_OK && n_m1 > 0) rc = run_batch1(problems, m1_idx, n_m1, st);
  if (rc == QTEA_OK && n_mb > 0) rc = run_mb(problems, mb_idx, n_mb, M, st);
  std::free(m1_idx);
  if (rc != QTEA_OK) cudaGetLastError();
  return rc;
}

int qtea_gemv_plan(const qtea_gemv_problem* problems, int n_problems, int M, int* kernels) {
  if (n_problems > 0 && !kernels) return QTEA_ERR_INVALID_ARG;
  int rc = check_call(problems, n_problems, M);
  if (rc) return rc;
  int m1_idx[kMaxProblems], n_m1 = 0;
  bool m1_many = false;
  for (int i = 0; i < n_problems; ++i) {
    switch (route(problems[i], M)) {
      case kRouteNone:
      case kRouteZero: kernels[i] = QTEA_KERNEL_NONE; break;
      case kRouteBatch1:
        kernels[i] = QTEA_KERNEL_STREAM_K;
        if (n_m1 < kMaxProblems) m1_idx[n_m1++] = i;
        else m1_many = true;
        break;
      case kRouteLut: kernels[i] = QTEA_KERNEL_LUT; break;
      case kRouteMb: kernels[i] = QTEA_KERNEL_LOW_BATCH; break;
      case kRouteB3: kernels[i] = QTEA_KERNEL_BASE3_FIXED; break;
      case kRoutePaper: kernels[i] = QTEA_KERNEL_PAPER; break;
      case kRouteGeneric: kernels[i] = QTEA_KERNEL_GENERIC; break;
    }
  }
  RowsLaunch L;
  if (!m1_many && n_m1 > 0 && rows_plan(problems, m1_idx, n_m1, L))
    for (int k = 0; k < n_m1; ++k) kernels[m1_idx[k]] = QTEA_KERNEL_ROWS;
  return QTEA_OK;
}

int qtea_rows_plan_shapes(const int* N, const int* K, const int* n_salient, int n, int sm_count, size_t smem_optin,
                          int* ctas, int* plan) {
  if (!N || !K || !n_salient || !plan || n < 1 || n > kMaxProblems || sm_count < 1) return QTEA_ERR_INVALID_ARG;
  long long NN[kMaxProblems];
  int nch[kMaxProblems], sal[kMaxProblems];
  for (int i = 0; i < n; ++i) {
    if (N[i] < 1 || K[i] < 1 || N[i] > (1 << 20) || K[i] > 65536 || n_salient[i] < 0 || n_salient[i] > K[i] ||
        (n_salient[i] > 0 && N[i] % 4))
      return QTEA_ERR_INVALID_ARG;
    NN[i] = N[i];
    nch[i] = (K[i] + kChunkCols - 1) / kChunkCols;  // a 2-bit layout's chunks (K padded to 64 columns)
    sal[i] = n_salient[i];
  }
  RowsShapePlan P;
  if (!rows_plan_shapes(NN, nch, sal, n, sm_count, smem_optin, P)) return QTEA_ERR_UNSUPPORTED;
  plan[0] = P.grid;
  plan[1] = P.rows_cap;
  plan[2] = P.wide ? 1 : 0;
  plan[3] = P.kparts;
  if (ctas)
    for (int i = 0; i < n; ++i) ctas[i] = P.cnt[i];
  return QTEA_OK;
}

int qtea_gemv(const uint16_t* x, const qtea_layout* l, const uint16_t* row_scale, const uint16_t* col_scale,
              const int32_t* salient_idx, const uint16_t* residual_vals, const uint8_t* residual_idx, float* y, int M,
              qtea_stream_t stream) {
  qtea_gemv_problem q;
  q.x = x;
  q.packed_ternary = l;
  q.row_scale = row_scale;
  q.col_scale = col_scale;
  q.salient_idx = salient_idx;
  q.residual_vals = residual_vals;
  q.residual_idx = residual_idx;
  q.y = y;
  return qtea_gemv_grouped(&q, 1, M, stream);
}

void qtea_free(qtea_layout* layout) { release(layout); }

int qtea_layout_describe(const qtea_layout* l, qtea_layout_desc* out) {
  if (!l || !out) return QTEA_ERR_INVALID_ARG;
  out->N = l->N;
  out->K = l->K;
  out->K_pad = l->K_pad;
  out->group_size = l->group_size;
  out->n_salient = l->n_salient;
  out->format = l->format;
  out->packed_bytes = l->packed_bytes;
  out->packed_data = l->packed;
  out->batch1_kernel = (l->m1_ok && m1_capable(l)) ? 1 : 0;
  out->rows_kernel = rows_capable(l) ? 1 : 0;
  out->options = l->options;
  return QTEA_OK;
}

int qtea_quantize(const float* W, const float* hdiag, int N, int K, int group_size, int n_salient, int options,
                  int fit_iters, int rescale_iters, int8_t* codes, uint16_t* row_scale, uint16_t* col_scale,
                  int32_t* salient_idx, uint16_t* residual_vals, uint8_t* residual_idx, qtea_stream_t stream) {
  if (N <= 0 || K <= 0 || N > (1 << 20) || K > 65536 || n_salient < 0 || n_salient > K) return QTEA_ERR_INVALID_ARG;
  if (group_size != K && group_size != 128) return QTEA_ERR_UNSUPPORTED;
  if (n_salient > 0 && N % 4 != 0) return QTEA_ERR_INVALID_ARG;
  if (options & ~QTEA_OPT_BIAS) return QTEA_ERR_INVALID_ARG;
  if (fit_iters < 0 || fit_iters > 64 || rescale_iters < 0 || rescale_iters > 64) return QTEA_ERR_INVALID_ARG;
  if (!W || !hdiag || !codes || !row_scale || !col_scale) return QTEA_ERR_INVALID_ARG;
  if (n_salient > 0 && (!salient_idx || !residual_vals || !residual_idx)) return QTEA_ERR_INVALID_ARG;
  if (!aligned(W, 4) || !aligned(hdiag, 4) || !aligned(row_scale, 2) || !aligned(col_scale, 2) ||
      (n_salient > 0 && (!aligned(salient_idx, 4) || !aligned(residual_vals, 2))))
    return QTEA_ERR_INVALID_ARG;
  QuantArgs a;
  a.W = W;
  a.h = hdiag;
  a.N = N;
  a.K = K;
  a.group = group_size;
  a.s = n_salient;
  a.bias = (options & QTEA_OPT_BIAS) ? 1 : 0;
  a.fit_iters = fit_iters;
  a.rescale_iters = rescale_iters;
  a.codes = codes;
  a.row_scale = row_scale;
  a.col_scale = col_scale;
  a.sal = salient_idx;
  a.rvals = residual_vals;
  a.ridx = residual_idx;
  if (launch_quantize(a, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  return QTEA_OK;
}

int qtea_set_layout_options(qtea_layout* l, int options) {
  if (!l || (options & ~(QTEA_OPT_BIAS | QTEA_OPT_RESIDUAL_FP8 | QTEA_OPT_FIXED_POINT | QTEA_OPT_STREAM_K)) != 0)
    return QTEA_ERR_INVALID_ARG;
  l->options = options;
  return QTEA_OK;
}

int qtea_set_activation_precision(qtea_layout* l, int bits) {
  if (!l || (bits != 16 && bits != 24)) return QTEA_ERR_INVALID_ARG;
  l->act_bits = bits;
  return QTEA_OK;
}

int qtea_salient_from_bitmap(const uint32_t* bitmap, int K, int32_t* salient_idx, int max_s, int* n_salient,
                             qtea_stream_t stream) {
  if (K < 0 || max_s < 0 || !n_salient || (K > 0 && (!bitmap || !aligned(bitmap, 4))) ||
      (max_s > 0 && (!salient_idx || !aligned(salient_idx, 4))))
    return QTEA_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int* count = nullptr;
  if (cudaMalloc(&count, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_ALLOC;
  }
  int host = 0;
  int rc = QTEA_OK;
  if (launch_bitmap_to_index(bitmap, K, salient_idx, max_s, count, st) != cudaSuccess ||
      cudaMemcpyAsync(&host, count, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    rc = QTEA_ERR_CUDA;
  cudaFree(count);
  if (rc != QTEA_OK) {
    cudaGetLastError();
    return rc;
  }
  *n_salient = host;
  return host > max_s ? QTEA_ERR_INVALID_ARG : QTEA_OK;
}

int qtea_salient_to_bitmap(const int32_t* salient_idx, int n_salient, int K, uint32_t* bitmap, qtea_stream_t stream) {
  if (K < 0 || n_salient < 0 || n_salient > K || (n_salient > 0 && (!salient_idx || !aligned(salient_idx, 4))) ||
      (K > 0 && (!bitmap || !aligned(bitmap, 4))))
    return QTEA_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int* bad = nullptr;
  if (cudaMalloc(&bad, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_ALLOC;
  }
  int host = 0;
  int rc = QTEA_OK;
  if (cudaMemsetAsync(bad, 0, sizeof(int), st) != cudaSuccess ||
      launch_index_to_bitmap(salient_idx, n_salient, K, bitmap, bad, st) != cudaSuccess ||
      cudaMemcpyAsync(&host, bad, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    rc = QTEA_ERR_CUDA;
  cudaFree(bad);
  if (rc != QTEA_OK) {
    cudaGetLastError();
    return rc;
  }
  return host ? QTEA_ERR_INVALID_ARG : QTEA_OK;
}

int qtea_layout_copy_packed(const qtea_layout* l, void* dst, size_t bytes, qtea_stream_t stream) {
  if (!l || bytes != l->packed_bytes || (bytes > 0 && !dst)) return QTEA_ERR_INVALID_ARG;
  if (bytes == 0) return QTEA_OK;
  if (cudaMemcpyAsync(dst, l->packed, bytes, cudaMemcpyDeviceToDevice, reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  return QTEA_OK;
}

int qtea_device_status(const qtea_layout* l, qtea_stream_t stream) {
  if (!l) return QTEA_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int flag = 0;
  if (cudaMemcpyAsync(&flag, l->status, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaMemsetAsync(l->status, 0, sizeof(int), st) != cudaSuccess || cudaStreamSynchronize(st) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  return flag == 0 ? QTEA_OK : flag;
}

int qtea_gemv_m1_static(const uint16_t* x, const uint8_t* packed, int N, int K, int n_salient,
                        const uint16_t* row_scale, const uint16_t* col_scale, const int32_t* salient_idx,
                        const uint16_t* residual_vals, const uint8_t* residual_idx, float* y, qtea_stream_t stream) {
  if (N < 0 || K < 0 || n_salient < 0 || n_salient > K) return QTEA_ERR_INVALID_ARG;
  if (n_salient > 0 && N % 4 != 0) return QTEA_ERR_INVALID_ARG;
  if ((long long)K + 63 > 0x7fffffffLL) return QTEA_ERR_INVALID_ARG;
  if ((N + kTileRows - 1) / kTileRows > kStaticTiles) return QTEA_ERR_SCRATCH_LIMIT;
  if (N == 0) return QTEA_OK;
  if (!y || !aligned(y, 4)) return QTEA_ERR_INVALID_ARG;
  if (K > 0 && (!packed || !aligned(packed, 16))) return QTEA_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (K == 0) {
    if (cudaMemsetAsync(y, 0, (size_t)N * sizeof(float), st) != cudaSuccess) {
      cudaGetLastError();
      return QTEA_ERR_CUDA;
    }
    return QTEA_OK;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kStaticMaxDevices) return QTEA_ERR_UNSUPPORTED;
  StaticDevice d;
  int rc = static_setup(dev, &d);
  if (rc) return rc;

  // A layout record on the host stack that borrows the caller's packed codes and points the
  // split-tile scratch at the static array; the planner and kernels below are the ones qtea_gemv uses.
  qtea_layout l;
  std::memset(&l, 0, sizeof(l));
  l.N = N;
  l.K = K;
  l.K_pad = round_up(K, 64);
  l.group_size = K;
  l.n_salient = n_salient;
  l.format = QTEA_FMT_2BIT;
  l.packed_bytes = (size_t)N * (size_t)(l.K_pad / 4);
  l.packed = const_cast<uint8_t*>(packed);
  l.device = dev;
  l.sm_count = d.sm_count;
  l.smem_optin = d.smem_optin;
  l.act_bits = 16;
  l.n_tiles = (N + kTileRows - 1) / kTileRows;
  l.n_chunks = (l.K_pad + kChunkCols - 1) / kChunkCols;
  l.workspace = reinterpret_cast<float*>(d.scratch);
  l.counters = reinterpret_cast<unsigned*>(d.scratch + kStaticWsBytes);
  l.status = reinterpret_cast<int*>(d.scratch + kStaticWsBytes + kStaticCtrBytes);
  l.m1_ok = false;
  if (d.m1_ok) {
    cuuint64_t dims[2] = {(cuuint64_t)(l.K_pad / 4), (cuuint64_t)N};
    cuuint64_t strides[1] = {(cuuint64_t)(l.K_pad / 4)};
    cuuint32_t box[2] = {(cuuint32_t)kChunkRowBytes, (cuuint32_t)kBoxRows};
    cuuint32_t estr[2] = {1, 1};
    l.m1_ok = get_encode_tiled()(&l.tmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, l.packed, dims, strides, box, estr,
                                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }

  qtea_gemv_problem q;
  q.x = x;
  q.packed_ternary = &l;
  q.row_scale = row_scale;
  q.col_scale = col_scale;
  q.salient_idx = salient_idx;
  q.residual_vals = residual_vals;
  q.residual_idx = residual_idx;
  q.y = y;
  rc = check_problem(q, 1);
  if (rc) return rc;
  const int idx0 = 0;
  rc = l.m1_ok ? run_m1(&q, &idx0, 1, st, true) : launch_generic_problem(q, 1, st);
  if (rc != QTEA_OK) cudaGetLastError();
  return rc;
}

int qtea_gemv_m1_static_status(int clear, qtea_stream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kStaticMaxDevices) return QTEA_ERR_UNSUPPORTED;
  StaticDevice d;
  int rc = static_setup(dev, &d);
  if (rc) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned char* ctr = d.scratch + kStaticWsBytes;  // counters, then the status word
  int* word = reinterpret_cast<int*>(d.scratch + kStaticWsBytes + kStaticCtrBytes);
  // host copies on this thread's stack (8 KB of counters): no allocation
  unsigned host_ctr[kStaticCtrBytes / sizeof(unsigned)];
  int host_word = 0;
  if (cudaMemcpyAsync(host_ctr, ctr, kStaticCtrBytes, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaMemcpyAsync(&host_word, word, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess) {
    cudaGetLastError();
    return QTEA_ERR_CUDA;
  }
  bool dirty = false;
  for (size_t k = 0; k < kStaticCtrBytes / sizeof(unsigned); ++k) dirty = dirty || host_ctr[k] != 0u;
  rc = host_word != 0 ? host_word : dirty ? QTEA_ERR_STATE : QTEA_OK;
  // partial rows, counters and status word back to zero: the start state of a call (a call that
  // timed out may have left partial rows that no CTA summed)
  if (clear && rc != QTEA_OK) {
    if (cudaMemsetAsync(d.scratch, 0, kStaticWsBytes + kStaticCtrBytes + sizeof(int), st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess) {
      cudaGetLastError();
      return QTEA_ERR_CUDA;
    }
  }
  return rc;
}

}  // extern "C"
