/*
 * qtea.h: C ABI of the GB300 (sm_103a) QTEA decode GEMV library.
 *
 * The operation is the inference-time product of the QTEA paper ("Ternary LLMs with
 * Sparse Residual Salient Weight and By-Column Optimization"):
 *
 *   y[m][o] = alpha[o] * sum_j T[o][j] * v[j] * x[m][j]                 (Sec. 3.5, Eq. 10)
 *           + sum_{c < s} [pos(o/4, c) == o % 4] * R[o/4][c] * x[m][S_c]  (Sec. 3.5, Eq. 11)
 *
 * i.e. y = x * W^T with the dequantized weight of Sec. 3.3, Eq. 4 (W^ = v_j * alpha_o * T_oj,
 * the bias beta being zero) plus the column-semi-sparse residual of Sec. 3.2 / Sec. 3.5: in
 * each salient column S_c, every group of four consecutive output rows holds exactly one
 * residual value and its 2-bit position inside the group (1:4 sparsity along the rows).
 * The paper's own storage is available too (Sec. 3.3 Eq. 4 and Sec. 3.5): alpha, and optionally
 * the bias beta, per row and group of 128 columns; base-3 codes; FP8 E4M3 residual values:
 *   y[m][o] = sum_g ( alpha[o][g] sum_{j in g} T v x + beta[o][g] sum_{j in g} x[m][j] ) + residual
 * (see qtea_pack_layout and qtea_set_layout_options).
 *
 * Conventions for every entry point:
 *   - fp16 tensors are IEEE 754 binary16 bit patterns passed as uint16_t.
 *   - All tensor pointers are DEVICE pointers owned by the caller, except the packed
 *     ternary weights, which the library owns inside a qtea_layout.
 *   - Arrays are dense and row-major. 16-byte alignment is required where stated.
 *   - Entry points return a qtea_status. Nothing is printed, no exception crosses the
 *     ABI, and there is no CPU fallback: without a usable GPU every call that computes
 *     fails with QTEA_ERR_CUDA.
 *   - `stream` is a cudaStream_t (0 = legacy default stream).
 */
#ifndef QTEA_H_
#define QTEA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* qtea_stream_t; /* identical to cudaStream_t */
typedef struct qtea_layout qtea_layout;    /* opaque, library-owned packed ternary weights */

typedef enum qtea_status {
  QTEA_OK = 0,
  QTEA_ERR_INVALID_ARG = 1, /* null pointer, negative or inconsistent size, misalignment */
  QTEA_ERR_BAD_CODES = 2,   /* a ternary code outside {-1, 0, +1} */
  QTEA_ERR_UNSUPPORTED = 3, /* a valid request this build does not implement */
  QTEA_ERR_CUDA = 4,        /* a CUDA runtime error (no device, launch failure, ...) */
  QTEA_ERR_ALLOC = 5,       /* device memory allocation failed */
  QTEA_ERR_TIMEOUT = 6,     /* a bounded wait inside a kernel gave up (see qtea_device_status) */
  QTEA_ERR_SCRATCH_LIMIT = 7, /* larger than the static scratch of qtea_gemv_m1_static allows */
  QTEA_ERR_STATE = 8          /* the static scratch of qtea_gemv_m1_static is not in its start state
                                 (see qtea_gemv_m1_static_status) */
} qtea_status;

typedef enum qtea_format {
  QTEA_FMT_2BIT = 0, /* 4 codes per byte, this library's layout */
  QTEA_FMT_BASE3 = 1 /* 5 codes per byte, 26 bytes per 128 columns: the paper's layout (Sec. 3.5) */
} qtea_format;

/* Layout options (qtea_set_layout_options), the paper's own storage of the scales and residual. */
typedef enum qtea_option {
  QTEA_OPT_BIAS = 1,         /* row_scale holds (alpha, beta) pairs: fp16 [N][G][2] (Eq. 4's beta) */
  QTEA_OPT_RESIDUAL_FP8 = 2, /* residual_vals holds FP8 E4M3 bytes [N/4][s] (Sec. 4.1), passed
                                through the same pointer argument */
  QTEA_OPT_FIXED_POINT = 4,  /* base-3 layouts: batch-1 calls decode by the fixed-point
                                dot-product kernel instead of the paper's sign-symmetric lookup
                                table (Sec. 3.5, Appendix A), the default */
  QTEA_OPT_STREAM_K = 8      /* 2-bit layouts: batch-1 calls always take the stream-K kernel, never
                                the row-resident one (see qtea_gemv_grouped) */
} qtea_option;

/* Largest batch (rows of x) one qtea_gemv call accepts. */
#define QTEA_MAX_M 16

/*
 * Pack ternary codes into the library's 2-bit layout (Sec. 3.1, Eq. 2 gives T; the layout is
 * this library's own, chosen for 16-byte coalesced loads).
 *
 *   ternary_codes  device int8 [N][K], values -1, 0, +1 (read only; may be freed afterwards)
 *   N, K           output rows and input columns, N >= 0, K >= 0
 *   group_size     K (one alpha per row) or 128 (alpha per row and group of 128 columns,
 *                  G = ceil(K/128) groups, the last one possibly shorter); anything else ->
 *                  QTEA_ERR_UNSUPPORTED
 *   n_salient      number of salient columns s the layout will be used with, s >= 0;
 *                  if s > 0, N must be a multiple of 4 (groups of four rows)
 *   format         QTEA_FMT_2BIT or QTEA_FMT_BASE3
 *   out            receives the new layout on success, NULL on failure
 *
 * Packed layout (2-bit): K_pad = K rounded up to a multiple of 64. Row r occupies bytes
 * [r*K_pad/4, (r+1)*K_pad/4); column k sits in byte r*K_pad/4 + k/4 at bits 2*(k%4) and
 * 2*(k%4)+1 (least significant first) as the code T+1; columns k >= K hold code 1.
 * Base-3 layout: K_pad = K rounded up to a multiple of 128; each row is K_pad/128 groups of 26
 * bytes; byte q of group h holds columns 128h + 5q + d, d = 0..4, as sum_d (T+1) 3^d (lowest
 * column in the least significant digit); byte 25 holds three columns and two pad digits; pad
 * digits and columns >= K are digit 1.
 * Which kernel serves a call: the TMA batch-1 kernel takes 2-bit layouts with fp16 residual values
 * at M = 1 (one alpha per row, or alpha and beta per row or per 128-column group), in one of two
 * forms: a row-resident launch, where every CTA holds all the codes of its rows at once (taken when
 * all of a call's batch-1 problems have one alpha per row, K <= 8192 and at most 512 salient
 * columns, and fit one such launch: at most 32 rows per CTA with one or two CTAs per SM, one when
 * some problem has K > 4096 or more than 256 salient columns;
 * a latency-bound form for small calls), else the persistent stream-K launch; the tensor-core
 * low-batch kernel takes those at M >= 2 and 2-bit layouts with FP8 residual values (groups of 128
 * columns, or beta absent) at any M; base-3 layouts
 * at M = 1 run on the paper's table-lookup decode (Sec. 3.5, Appendix A); base-3 layouts at
 * 2 <= M <= 4 (or at M = 1 with QTEA_OPT_FIXED_POINT) run on a kernel that stages v*x once per CTA
 * in fixed point (the base-3 problems of a grouped call share one launch); the rest run on general
 * kernels.
 *
 * The call validates every code on the device and synchronizes `stream` once to read the
 * result; invalid codes give QTEA_ERR_BAD_CODES and no layout. It allocates the packed
 * bytes and the split-K workspace of qtea_gemv (both freed by qtea_free).
 */
int qtea_pack_layout(const int8_t* ternary_codes, int N, int K, int group_size, int n_salient, int format,
                     qtea_stream_t stream, qtea_layout** out);

/*
 * y = x * W^T for the layout's N x K ternary weights plus the 1:4 salient residual
 * (Eq. 10 and Eq. 11: one alpha per row, or alpha and optionally beta per row and group of 128
 * columns as the layout's group_size and options say).
 *
 *   x              device fp16 [M][K], activations
 *   packed_ternary layout from qtea_pack_layout
 *   row_scale      device fp16 [N][G], alpha (G = 1 unless the layout's group_size is 128);
 *                  with QTEA_OPT_BIAS, [N][G][2]: alpha then beta of each group
 *   col_scale      device fp16 [K], v_j, the column-wise rescale factors (Sec. 3.3, Eq. 4)
 *   salient_idx    device int32 [s], strictly ascending column indices, each in [0, K)
 *   residual_vals  device fp16 [N/4][s]: R of group q (rows 4q..4q+3) in salient column c
 *                  (FP8 E4M3 bytes [N/4][s] with QTEA_OPT_RESIDUAL_FP8)
 *   residual_idx   device uint8 [N/4][ceil(s/4)]: 2-bit position of that value in its
 *                  group; entry (q, c) at bits 2*(c%4) of byte q*ceil(s/4) + c/4
 *   y              device fp32 [M][N], overwritten
 *   M              batch, 1 <= M <= QTEA_MAX_M
 *   stream         CUDA stream; the call is asynchronous and allocates nothing
 *
 * s is the layout's n_salient; with s = 0 the three residual pointers may be NULL.
 * Alignment: fp16 arrays 2 bytes, salient_idx and y 4 bytes. The salient indices are
 * not validated on the device: out-of-order or duplicate indices give an unspecified y
 * (each listed column's residual is still added once), indices outside [0, K) are
 * clamped into range and never read out of bounds.
 * Calls that share a layout must be ordered on one stream: the layout holds the split-K
 * workspace. Results are bitwise reproducible for a given (layout, inputs, device); a grouped
 * call (qtea_gemv_grouped) is reproducible for the same group, but its rounding may differ
 * from separate calls because the split of work over the CTAs differs.
 * Numerics: at M = 1 (the library's own storage) the ternary sum is accumulated exactly in
 * integers over 512-column blocks, with v*x represented in 16-bit or 24-bit fixed point relative
 * to the block's largest |v*x| after its massive values are taken out and added exactly in fp32
 * (qtea_set_activation_precision); block sums, alpha and the residual are combined in fp32. At 2 <= M <= 16, and for 2-bit layouts in the paper's
 * storage at any M, the tensor cores take 2T*v and x in fp16 (both exact, which needs |v| < 32768)
 * with exact fp32 products and fp32 sums; alpha, beta and the residual are applied in fp32.
 * Base-3 layouts at M <= 4 (when v*x of the call fits in shared memory): the ternary sum is
 * accumulated exactly in integers over 128-column blocks, with v*x in fixed point relative to the
 * block's largest |v*x| (|X| < 2^23) after up to 3 massive values per block are taken out and
 * added exactly in fp32; block sums, alpha, beta and the residual are combined in fp32. Other
 * layouts and batch sizes: fp32 throughout.
 */
int qtea_gemv(const uint16_t* x, const qtea_layout* packed_ternary, const uint16_t* row_scale,
              const uint16_t* col_scale, const int32_t* salient_idx, const uint16_t* residual_vals,
              const uint8_t* residual_idx, float* y, int M, qtea_stream_t stream);

/* One GEMV of a grouped call: the arguments of qtea_gemv except M and the stream. */
typedef struct qtea_gemv_problem {
  const uint16_t* x;
  const qtea_layout* packed_ternary;
  const uint16_t* row_scale;
  const uint16_t* col_scale;
  const int32_t* salient_idx;
  const uint16_t* residual_vals;
  const uint8_t* residual_idx;
  float* y;
} qtea_gemv_problem;

/*
 * Several independent GEMVs with the same batch M, as if qtea_gemv were called for each in
 * order, but sharing launches: up to 8 consecutive problems that the same kernel variant serves
 * (batch 1; low batch with one alpha per row; low batch with scale groups) run in one persistent
 * launch, which removes per-launch ramp-up and tail time when the problems are small (e.g. the
 * q/k/v/o/gate/up/down GEMVs of one decoder layer).
 * Every problem is validated before anything is launched; a failing check returns its status
 * and launches nothing. No two problems may write overlapping y, and problems must not share
 * a layout. QTEA_ERR_TIMEOUT from a grouped launch is recorded in the layout of the first
 * problem of that launch (qtea_device_status). The call is asynchronous on `stream`.
 */
int qtea_gemv_grouped(const qtea_gemv_problem* problems, int n_problems, int M, qtea_stream_t stream);

/* The kernels that serve problems (see "Which kernel serves a call" at qtea_pack_layout). */
typedef enum qtea_kernel {
  QTEA_KERNEL_NONE = 0,         /* N = 0 (nothing to do) or K = 0 (y is zero-filled) */
  QTEA_KERNEL_ROWS = 1,         /* batch-1, row-resident launch */
  QTEA_KERNEL_STREAM_K = 2,     /* batch-1, persistent stream-K launch */
  QTEA_KERNEL_LUT = 3,          /* the paper's table-lookup decode (base-3 codes, M = 1) */
  QTEA_KERNEL_LOW_BATCH = 4,    /* tensor-core low-batch kernel (2-bit codes) */
  QTEA_KERNEL_BASE3_FIXED = 5,  /* base-3 codes, v*x staged once per CTA in fixed point */
  QTEA_KERNEL_PAPER = 6,        /* general kernel for the paper's storage */
  QTEA_KERNEL_GENERIC = 7       /* general kernel */
} qtea_kernel;

/*
 * The kernel that qtea_gemv_grouped(problems, n_problems, M, ...) would run for each problem:
 * kernels[i] receives a qtea_kernel value for problems[i]. Host-side only: no device work, no
 * synchronization. Arguments are validated as qtea_gemv_grouped validates them (same status
 * codes); kernels is a host array of n_problems ints, unchanged on error.
 */
int qtea_gemv_plan(const qtea_gemv_problem* problems, int n_problems, int M, int* kernels);

/*
 * The row-resident launch that qtea_gemv_grouped would plan for n batch-1 problems (2-bit codes,
 * one alpha per row, fp16 residual values) from their shapes alone (no counterpart in the paper:
 * it exposes the batch-1 dispatch rule so that it can be checked without a device). Problem i has
 * N[i] rows, K[i] columns and n_salient[i] salient columns; the device has sm_count SMs and
 * smem_optin bytes of opt-in shared memory per block (cudaDeviceProp::sharedMemPerBlockOptin).
 *   QTEA_OK               the problems fit one row-resident launch: plan[0..3] receive the grid
 *                         (CTAs), the most rows of a CTA, wide (1: K above 4096 or more than 256
 *                         salient columns somewhere, one CTA per SM) and the lanes per row of every
 *                         CTA (4, 2 or 1; 0 when the CTAs differ); ctas[i], when ctas is not NULL,
 *                         problem i's CTAs;
 *   QTEA_ERR_UNSUPPORTED  they take the stream-K launch (plan and ctas unchanged);
 *   QTEA_ERR_INVALID_ARG  a NULL array, n outside 1..8, sm_count < 1, N or K zero (such problems
 *                         launch nothing) or a shape qtea_pack_layout rejects.
 * Host only: touches no device.
 */
int qtea_rows_plan_shapes(const int* N, const int* K, const int* n_salient, int n, int sm_count,
                          size_t smem_optin, int* ctas, int* plan);

/* Release a layout and its device memory. NULL is ignored. The caller orders it after the
 * last qtea_gemv that uses the layout has completed; it synchronizes nothing itself. */
void qtea_free(qtea_layout* layout);

/*
 * The quantizer's per-layer steps (Sec. 3.1-3.3 and the 1:4 residual of Sec. 3.2 / 3.5; not the
 * error propagation of Sec. 3.4), from full-precision weights to this library's inputs:
 *
 *   W              device fp32 [N][K], the full-precision weights (row = output feature)
 *   hdiag          device fp32 [K], diag(H) of the calibration Hessian (Sec. 3.2)
 *   group_size     K (one alpha per row) or 128 (alpha, and beta with QTEA_OPT_BIAS, per group)
 *   n_salient      s, 0 <= s <= K; N % 4 == 0 when s > 0
 *   options        0 or QTEA_OPT_BIAS (beta = the group mean; without it beta = 0)
 *   fit_iters      refits of alpha as the mean |W - beta| over the nonzero codes (0 .. 64)
 *   rescale_iters  rounds of the column rescale v_j and reassignment (0 .. 64; the paper uses a
 *                  small number, e.g. 2)
 *   codes          out: device int8 [N][K], T in {-1, 0, +1} (the input of qtea_pack_layout)
 *   row_scale      out: device fp16 [N][G] alpha, or [N][G][2] (alpha, beta) with QTEA_OPT_BIAS
 *   col_scale      out: device fp16 [K] v
 *   salient_idx    out: device int32 [s], ascending: the s columns with the largest
 *                  max_i W_ij^2 hdiag_j^2 (ties: lower column)
 *   residual_vals  out: device fp16 [N/4][s], residual_idx out: device uint8 [N/4][ceil(s/4)]: per
 *                  group of four rows and salient column, the largest W - W^ and its position
 *
 * Decisions are taken in fp32 with every sum in index order, so the outputs are reproducible bit
 * for bit. Asynchronous on `stream`; scratch (about 16 K + 8 N G bytes) comes from the
 * stream-ordered allocator.
 * Limits: 1 <= N <= 2^20, 1 <= K <= 65536; W and hdiag 4-byte aligned, row_scale, col_scale and
 * residual_vals 2-byte aligned, salient_idx 4-byte aligned. Returns QTEA_ERR_INVALID_ARG or
 * QTEA_ERR_UNSUPPORTED for arguments outside the above, QTEA_ERR_CUDA when a launch or the
 * scratch allocation fails.
 */
int qtea_quantize(const float* W, const float* hdiag, int N, int K, int group_size, int n_salient, int options,
                  int fit_iters, int rescale_iters, int8_t* codes, uint16_t* row_scale, uint16_t* col_scale,
                  int32_t* salient_idx, uint16_t* residual_vals, uint8_t* residual_idx, qtea_stream_t stream);

/* Static English description of a status code. Never NULL. */
const char* qtea_status_string(int status);

/* Read-only description of a layout (all sizes in elements unless named *_bytes). */
typedef struct qtea_layout_desc {
  int N, K, K_pad, group_size, n_salient, format;
  size_t packed_bytes;      /* size of the packed ternary weights */
  const void* packed_data;  /* device pointer to the packed ternary weights */
  int batch1_kernel;        /* 1 if M = 1 calls run the TMA stream-K batch-1 kernel (2-bit codes,
                               fp16 residual values), 0 otherwise */
  int options;              /* QTEA_OPT_* flags */
  int rows_kernel;          /* 1 if M = 1 calls may run the row-resident kernel instead (2-bit codes,
                               one alpha per row, fp16 residual values, K <= 8192, n_salient <= 512,
                               no QTEA_OPT_STREAM_K): they do when all of a call's batch-1 problems
                               fit one launch of it */
} qtea_layout_desc;

int qtea_layout_describe(const qtea_layout* layout, qtea_layout_desc* out);

/*
 * The salient set as the paper stores it (Sec. 3.5: a binary bitmap over the input columns) and as
 * qtea_gemv takes it (salient_idx: int32, strictly ascending, each < K).
 *   bitmap     device uint32 [ceil(K/32)]: column j is bit j % 32 (least significant first) of
 *              word j / 32; bits of columns >= K are ignored by qtea_salient_from_bitmap and zero
 *              after qtea_salient_to_bitmap
 *   salient_idx  device int32 [max_s] (written) / [n_salient] (read)
 * qtea_salient_from_bitmap writes the marked columns in ascending order and their number to
 * *n_salient (host memory); more than max_s marked columns: QTEA_ERR_INVALID_ARG, *n_salient = the
 * number, the first max_s written. qtea_salient_to_bitmap overwrites the whole bitmap; an index
 * outside [0, K) or not above its predecessor gives QTEA_ERR_INVALID_ARG (the bitmap then holds the
 * valid ones). Both run on `stream`, synchronize it once, and allocate a 4-byte device word for the
 * duration of the call (setup-time utilities, not for the decode loop). Null or misaligned pointers,
 * K < 0 or max_s < 0: QTEA_ERR_INVALID_ARG.
 */
int qtea_salient_from_bitmap(const uint32_t* bitmap, int K, int32_t* salient_idx, int max_s, int* n_salient,
                             qtea_stream_t stream);
int qtea_salient_to_bitmap(const int32_t* salient_idx, int n_salient, int K, uint32_t* bitmap, qtea_stream_t stream);

/* Copy the layout's packed ternary bytes (qtea_layout_desc.packed_bytes of them) to the
 * caller's device buffer `dst`, asynchronously on `stream`. `bytes` must equal packed_bytes. */
int qtea_layout_copy_packed(const qtea_layout* layout, void* dst, size_t bytes, qtea_stream_t stream);

/*
 * Activation precision of batch-1 (M = 1) calls on this layout. The ternary sum is always
 * accumulated exactly in integers over 512-column blocks; what changes is how finely v*x is
 * represented in fixed point. In each block, values at least 16 times larger than all the others
 * (up to 16 of them, e.g. an LLM's massive activations) are taken out and added exactly in fp32;
 * the rest are held relative to their largest magnitude:
 *   bits = 16 (default): 16-bit (|X| < 2^15, two byte planes) for every block whose remaining
 *              largest |v*x| is at most 8 times their root mean square; other blocks, and
 *              layouts with K < 1024, use 24 bits.
 *   bits = 24: 24-bit (|X| < 2^23, three byte planes, half again as many dot-product
 *              instructions per weight) for every block.
 * Returns QTEA_ERR_INVALID_ARG for other values. Batch sizes M > 1 are not affected.
 */
int qtea_set_activation_precision(qtea_layout* layout, int bits);

/*
 * Storage options of the scales and residual values qtea_gemv reads with this layout: any
 * combination of QTEA_OPT_BIAS and QTEA_OPT_RESIDUAL_FP8 (0 restores fp16 alpha only and fp16
 * residual values), and QTEA_OPT_FIXED_POINT for base-3 layouts (at M = 1 base-3 layouts decode by
 * table lookup unless this option asks for the fixed-point kernel; at 2 <= M <= 4 they always use
 * the fixed-point kernel). Other bits -> QTEA_ERR_INVALID_ARG.
 * With QTEA_OPT_BIAS or QTEA_OPT_RESIDUAL_FP8 set, calls leave the batch-1 kernel (see
 * qtea_pack_layout for which kernel serves which storage); QTEA_OPT_FIXED_POINT changes nothing for
 * 2-bit layouts. Set it before the calls that use it; it takes effect for calls made afterwards.
 */
int qtea_set_layout_options(qtea_layout* layout, int options);

/*
 * Status written by the kernels of this layout: QTEA_OK, or QTEA_ERR_TIMEOUT if a bounded
 * wait inside a kernel gave up (the kernel then skipped its remaining work and y is
 * unspecified; the layout's split-tile workspace may then hold partial rows that no CTA summed,
 * so later calls on the layout are unspecified too: free it and pack a new one). Synchronizes
 * `stream`, reads the flag and clears it.
 */
int qtea_device_status(const qtea_layout* layout, qtea_stream_t stream);

/*
 * Allocation-free batch-1 GEMV. The QTEA paper has no counterpart: this is a deployment entry
 * point of this library, not a step of the method.
 *
 * Some callers cannot call cudaMalloc: a serving process whose allocator has already reserved the
 * GPU's memory for its own pool (a further cudaMalloc fails or escapes its accounting), or code on
 * a latency-critical path where cudaMalloc and cudaFree may synchronise the device. qtea_gemv needs
 * a qtea_layout, whose creation allocates. This call instead reads the packed codes from memory the
 * caller owns and takes its split-tile scratch from a fixed array in the library's static device
 * memory. It calls no cudaMalloc, cudaFree or other allocating routine.
 *
 * Computes what qtea_gemv computes for M = 1 on a layout with one alpha per row, no beta and fp16
 * residual values, with the default activation precision (qtea_set_activation_precision).
 *   x, row_scale, col_scale, salient_idx, residual_vals, residual_idx, y
 *                  as for qtea_gemv, with M = 1
 *   packed         device, 16-byte aligned, caller-owned: the 2-bit layout qtea_pack_layout
 *                  writes, N rows of K_pad/4 bytes (K_pad = K rounded up to a multiple of 64),
 *                  code T+1 four per byte, least significant first, pad columns code 1 (for
 *                  instance a copy made once with qtea_layout_copy_packed). Codes are not
 *                  validated: code 3 decodes as T = 2. The call's kernel reads them only after the
 *                  preceding work on `stream` has completed, so a kernel that writes them just
 *                  before the call on the same stream is seen.
 *   N, K, n_salient  sizes as for qtea_pack_layout (N % 4 == 0 when n_salient > 0)
 * Limits of the static scratch (663,808 bytes of device memory per device): N <= 131072 (at most
 * 256 tiles of 512 rows); a larger N returns QTEA_ERR_SCRATCH_LIMIT. At most 160 CTAs are used.
 * Set-up: the first call on each device, with that device current, looks the scratch up with
 * cudaGetSymbolAddress and sets the kernel's shared-memory attribute. Make that first call before
 * any stream capture on the device. Later calls encode a tensor map on the host and launch.
 * Start state: the split-tile partial rows, counters and the status word in the scratch must be
 * zero when a call starts. Static device memory is zero when the library's module loads, and every
 * completed call leaves them at zero. A call whose kernel gave up a bounded wait (QTEA_ERR_TIMEOUT)
 * can leave partial rows set: qtea_gemv_m1_static_status reports the timeout and, with clear,
 * restores the start state.
 * Concurrency: every call on a device shares the one scratch. Calls that may overlap on the
 * device (different streams without ordering, several host threads) race and give wrong results:
 * order them, e.g. on one stream.
 * Returns QTEA_OK, QTEA_ERR_INVALID_ARG, QTEA_ERR_SCRATCH_LIMIT, QTEA_ERR_UNSUPPORTED (device
 * ordinal >= 64) or QTEA_ERR_CUDA. A timeout inside the kernel is not reported by this call (it
 * is asynchronous): qtea_gemv_m1_static_status reads it.
 */
int qtea_gemv_m1_static(const uint16_t* x, const uint8_t* packed, int N, int K, int n_salient,
                        const uint16_t* row_scale, const uint16_t* col_scale, const int32_t* salient_idx,
                        const uint16_t* residual_vals, const uint8_t* residual_idx, float* y,
                        qtea_stream_t stream);

/*
 * State of the static scratch of qtea_gemv_m1_static on the current device (no counterpart in the
 * paper; it serves the allocation-free entry point). Synchronizes `stream`, then reads the
 * scratch's status word and split-tile counters:
 *   QTEA_OK           both at zero;
 *   QTEA_ERR_TIMEOUT  a kernel of an earlier call gave up a bounded wait (its y is unspecified, and
 *                     partial rows it left in the scratch would corrupt later calls);
 *   QTEA_ERR_STATE    counters left set without a recorded timeout.
 * With clear != 0, a non-OK state is reset to zero afterwards (partial rows, counters and status
 * word: cudaMemsetAsync on the static array, then a synchronization of `stream`), so the next call
 * starts correctly. Order this call after the calls it inspects, e.g. on the same stream. It
 * allocates nothing (the counters are copied to an 8 KB array on the calling thread's stack).
 * Returns the state above, or QTEA_ERR_UNSUPPORTED (device ordinal >= 64) or QTEA_ERR_CUDA.
 */
int qtea_gemv_m1_static_status(int clear, qtea_stream_t stream);

/*
 * Diagnostic, not a step of the GEMV (the paper has no counterpart): the issue rates that decide
 * between a dp4a decode and a tensor-core (mma.sync) decode of the 2-bit codes at batch 1, measured
 * on the current device, in clock cycles per instruction per SM sub-partition (8 warps per SM, 8
 * independent accumulator chains per warp):
 *   [0] mma.sync m16n8k16 f16 -> f32, constant operands
 *   [1] the same with A masked from a word that changes every instruction (as a decode builds it)
 *   [2] mma.sync m16n8k32 e4m3 -> f32, constant operands
 *   [3] the same with A masked from a changing word
 *   [4] dp4a
 *   cycles_per_instruction  host array of n >= 5 doubles, written
 * Allocates a few kilobytes of device memory and synchronizes the device. Returns QTEA_OK,
 * QTEA_ERR_INVALID_ARG (null array or n < 5), QTEA_ERR_ALLOC or QTEA_ERR_CUDA.
 */
int qtea_probe_decode_rates(double* cycles_per_instruction, int n);

#ifdef __cplusplus
}
#endif

#endif /* QTEA_H_ */
