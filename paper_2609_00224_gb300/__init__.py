"""Python binding of the QTEA GB300 GEMV library (``libqtea.so``, C ABI in ``include/qtea.h``).

The functions here have the C entry points' names and only marshal arguments: they check
dtypes and shapes of torch CUDA tensors, pass raw device pointers and the current CUDA
stream, and raise ``QteaError`` on a non-zero status. Every step of the computation runs in
the library's kernels; there is no fallback: if the library cannot be built or loaded, or
no GPU is present, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

from . import build as _build

QTEA_OK = 0
QTEA_ERR_INVALID_ARG = 1
QTEA_ERR_BAD_CODES = 2
QTEA_ERR_UNSUPPORTED = 3
QTEA_ERR_CUDA = 4
QTEA_ERR_ALLOC = 5
QTEA_ERR_TIMEOUT = 6
QTEA_ERR_SCRATCH_LIMIT = 7
QTEA_ERR_STATE = 8
QTEA_FMT_2BIT = 0
QTEA_FMT_BASE3 = 1
QTEA_OPT_BIAS = 1
QTEA_OPT_RESIDUAL_FP8 = 2
QTEA_OPT_FIXED_POINT = 4
QTEA_OPT_STREAM_K = 8
QTEA_MAX_M = 16

_lib = None


class QteaError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {status_string(status)} (status {status})")
        self.status = status


class _Problem(ctypes.Structure):
    _fields_ = [("x", ctypes.c_void_p), ("packed_ternary", ctypes.c_void_p), ("row_scale", ctypes.c_void_p),
                ("col_scale", ctypes.c_void_p), ("salient_idx", ctypes.c_void_p), ("residual_vals", ctypes.c_void_p),
                ("residual_idx", ctypes.c_void_p), ("y", ctypes.c_void_p)]


class _LayoutDesc(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int), ("K", ctypes.c_int), ("K_pad", ctypes.c_int), ("group_size", ctypes.c_int),
                ("n_salient", ctypes.c_int), ("format", ctypes.c_int), ("packed_bytes", ctypes.c_size_t),
                ("packed_data", ctypes.c_void_p), ("batch1_kernel", ctypes.c_int), ("options", ctypes.c_int),
                ("rows_kernel", ctypes.c_int)]


def library_path() -> str:
    return _build.LIB_PATH


def load(build_if_missing: bool = True):
    """Load libqtea.so (compiling it first if it is missing or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.build() if build_if_missing else _build.LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"QTEA CUDA library not found at {path}; run paper_2609_00224_gb300/build.py")
    lib = ctypes.CDLL(path)
    P, i32 = ctypes.c_void_p, ctypes.c_int
    lib.qtea_pack_layout.restype = i32
    lib.qtea_pack_layout.argtypes = [P, i32, i32, i32, i32, i32, P, ctypes.POINTER(P)]
    lib.qtea_gemv.restype = i32
    lib.qtea_gemv.argtypes = [P, P, P, P, P, P, P, P, i32, P]
    lib.qtea_free.restype = None
    lib.qtea_free.argtypes = [P]
    lib.qtea_status_string.restype = ctypes.c_char_p
    lib.qtea_status_string.argtypes = [i32]
    lib.qtea_layout_describe.restype = i32
    lib.qtea_layout_describe.argtypes = [P, ctypes.POINTER(_LayoutDesc)]
    lib.qtea_device_status.restype = i32
    lib.qtea_device_status.argtypes = [P, P]
    lib.qtea_gemv_grouped.restype = i32
    lib.qtea_gemv_grouped.argtypes = [P, i32, i32, P]
    lib.qtea_gemv_plan.restype = i32
    lib.qtea_gemv_plan.argtypes = [P, i32, i32, P]
    lib.qtea_rows_plan_shapes.restype = i32
    lib.qtea_rows_plan_shapes.argtypes = [P, P, P, i32, i32, ctypes.c_size_t, P, P]
    lib.qtea_set_activation_precision.restype = i32
    lib.qtea_set_activation_precision.argtypes = [P, i32]
    lib.qtea_set_layout_options.restype = i32
    lib.qtea_set_layout_options.argtypes = [P, i32]
    lib.qtea_layout_copy_packed.restype = i32
    lib.qtea_layout_copy_packed.argtypes = [P, P, ctypes.c_size_t, P]
    lib.qtea_salient_from_bitmap.restype = i32
    lib.qtea_salient_from_bitmap.argtypes = [P, i32, P, i32, ctypes.POINTER(i32), P]
    lib.qtea_salient_to_bitmap.restype = i32
    lib.qtea_salient_to_bitmap.argtypes = [P, i32, i32, P, P]
    lib.qtea_gemv_m1_static.restype = i32
    lib.qtea_gemv_m1_static.argtypes = [P, P, i32, i32, i32, P, P, P, P, P, P, P]
    lib.qtea_gemv_m1_static_status.restype = i32
    lib.qtea_gemv_m1_static_status.argtypes = [i32, P]
    lib.qtea_quantize.restype = i32
    lib.qtea_quantize.argtypes = [P, P, i32, i32, i32, i32, i32, i32, i32, P, P, P, P, P, P, P]
    lib.qtea_probe_decode_rates.restype = i32
    lib.qtea_probe_decode_rates.argtypes = [P, i32]
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().qtea_status_string(int(status)).decode()


def _stream(stream) -> Optional[int]:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t, dtypes, name, shape=None):
    import torch
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype not in dtypes:
        raise TypeError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t.data_ptr()


def _f16_types():
    import torch
    return (torch.float16, torch.int16) + ((torch.uint16,) if hasattr(torch, "uint16") else ())


class Layout:
    """Owner of a qtea_layout handle (packed ternary weights + split-K workspace)."""

    def __init__(self, handle: int, N: int, K: int, n_salient: int, group_size: Optional[int] = None):
        self._h = ctypes.c_void_p(handle)
        self.N, self.K, self.n_salient = N, K, n_salient
        self.group_size = K if group_size is None else group_size
        self.options = 0

    @property
    def G(self) -> int:
        g = self.group_size or 1
        return (self.K + g - 1) // g if self.K else 1

    @property
    def handle(self):
        if not self._h:
            raise ValueError("layout was freed")
        return self._h

    def describe(self) -> dict:
        d = _LayoutDesc()
        rc = load().qtea_layout_describe(self.handle, ctypes.byref(d))
        if rc:
            raise QteaError(rc, "qtea_layout_describe")
        return {f: getattr(d, f) for f, _ in _LayoutDesc._fields_}

    def set_activation_precision(self, bits: int):
        """24 (default, exact to 24-bit fixed point) or 16 (fast mode for outlier-free blocks)."""
        rc = load().qtea_set_activation_precision(self.handle, int(bits))
        if rc:
            raise QteaError(rc, "qtea_set_activation_precision")
        return self

    def set_options(self, options: int):
        """QTEA_OPT_BIAS and/or QTEA_OPT_RESIDUAL_FP8: the paper's storage of beta and residual values."""
        rc = load().qtea_set_layout_options(self.handle, int(options))
        if rc:
            raise QteaError(rc, "qtea_set_layout_options")
        self.options = int(options)
        return self

    def free(self):
        if self._h:
            load().qtea_free(self._h)
            self._h = ctypes.c_void_p(None)

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def qtea_pack_layout(codes, n_salient: int = 0, group_size: Optional[int] = None, fmt: int = QTEA_FMT_2BIT,
                     stream=None) -> Layout:
    """Pack int8 ternary codes [N][K] (CUDA tensor) into a library-owned layout."""
    import torch
    if codes.dim() != 2:
        raise ValueError("codes must be [N][K]")
    N, K = codes.shape
    ptr = _ptr(codes, (torch.int8,), "codes")
    out = ctypes.c_void_p()
    rc = load().qtea_pack_layout(ptr, N, K, K if group_size is None else group_size, n_salient, fmt,
                                 _stream(stream), ctypes.byref(out))
    if rc:
        raise QteaError(rc, "qtea_pack_layout")
    return Layout(out.value, N, K, n_salient, K if group_size is None else group_size)


def _problem_args(x, layout, row_scale, col_scale, salient_idx, residual_vals, residual_idx, y):
    import torch
    f16 = _f16_types()
    if x.dim() != 2:
        raise ValueError("x must be [M][K]")
    M = x.shape[0]
    N, K, s = layout.N, layout.K, layout.n_salient
    if y is None:
        y = torch.empty((M, N), dtype=torch.float32, device=x.device)
    args = [
        _ptr(x, f16, "x", (M, K)),
        layout.handle,
        _ptr(row_scale.reshape(-1) if row_scale is not None else None, f16, "row_scale",
             (N * layout.G * (2 if layout.options & QTEA_OPT_BIAS else 1),)),
        _ptr(col_scale, f16, "col_scale", (K,)),
        _ptr(salient_idx, (torch.int32,), "salient_idx", (s,)) if s else None,
        _ptr(residual_vals, (torch.uint8,) if layout.options & QTEA_OPT_RESIDUAL_FP8 else f16, "residual_vals",
             (N // 4, s)) if s else None,
        _ptr(residual_idx, (torch.uint8,), "residual_idx", (N // 4, (s + 3) // 4)) if s else None,
        _ptr(y, (torch.float32,), "y", (M, N)),
    ]
    return args, y, M


def qtea_gemv(x, layout: Layout, row_scale, col_scale, salient_idx=None, residual_vals=None, residual_idx=None,
              y=None, stream=None):
    """y[M][N] = x[M][K] * W^T (fp32) with the layout's ternary weights and the 1:4 residual."""
    args, y, M = _problem_args(x, layout, row_scale, col_scale, salient_idx, residual_vals, residual_idx, y)
    rc = load().qtea_gemv(*args, M, _stream(stream))
    if rc:
        raise QteaError(rc, "qtea_gemv")
    return y


def _problem_array(problems):
    ys, arr, M = [], (_Problem * max(len(problems), 1))(), None
    for i, q in enumerate(problems):
        args, y, m = _problem_args(q["x"], q["layout"], q["row_scale"], q["col_scale"], q.get("salient_idx"),
                                   q.get("residual_vals"), q.get("residual_idx"), q.get("y"))
        if M is None:
            M = m
        elif m != M:
            raise ValueError("all problems of a grouped call need the same batch M")
        args[1] = args[1].value
        arr[i] = _Problem(*args)
        ys.append(y)
    return arr, ys, M or 1


def qtea_gemv_grouped(problems, stream=None):
    """Several independent GEMVs in as few launches as possible.

    `problems` is a sequence of dicts with keys x, layout, row_scale, col_scale and optionally
    salient_idx, residual_vals, residual_idx, y. Returns the list of y tensors.
    """
    arr, ys, M = _problem_array(problems)
    rc = load().qtea_gemv_grouped(ctypes.cast(arr, ctypes.c_void_p), len(problems), M, _stream(stream))
    if rc:
        raise QteaError(rc, "qtea_gemv_grouped")
    return ys


QTEA_KERNEL_NAMES = {0: "none", 1: "rows", 2: "stream_k", 3: "lut", 4: "low_batch", 5: "base3_fixed", 6: "paper",
                     7: "generic"}


def qtea_gemv_plan(problems) -> list:
    """The kernel qtea_gemv_grouped(problems) would run for each problem, by name (QTEA_KERNEL_NAMES)."""
    arr, _, M = _problem_array(problems)
    out = (ctypes.c_int * max(len(problems), 1))()
    rc = load().qtea_gemv_plan(ctypes.cast(arr, ctypes.c_void_p), len(problems), M, ctypes.cast(out, ctypes.c_void_p))
    if rc:
        raise QteaError(rc, "qtea_gemv_plan")
    return [QTEA_KERNEL_NAMES[out[i]] for i in range(len(problems))]


def qtea_rows_plan_shapes(shapes, sm_count: int, smem_optin: int):
    """The row-resident launch qtea_gemv_grouped would plan for batch-1 problems of these (N, K,
    n_salient) shapes on a device of sm_count SMs (host only): a dict with grid, rows_cap, wide,
    kparts and ctas (per problem), or None when they take the stream-K launch."""
    n = len(shapes)
    arr = lambda vals: (ctypes.c_int * max(n, 1))(*vals)
    N, K, S = arr([int(a) for a, _, _ in shapes]), arr([int(b) for _, b, _ in shapes]), arr([int(c) for _, _, c in shapes])
    ctas, plan = (ctypes.c_int * max(n, 1))(), (ctypes.c_int * 4)()
    rc = load().qtea_rows_plan_shapes(ctypes.cast(N, ctypes.c_void_p), ctypes.cast(K, ctypes.c_void_p),
                                      ctypes.cast(S, ctypes.c_void_p), n, int(sm_count), int(smem_optin),
                                      ctypes.cast(ctas, ctypes.c_void_p), ctypes.cast(plan, ctypes.c_void_p))
    if rc == QTEA_ERR_UNSUPPORTED:
        return None
    if rc:
        raise QteaError(rc, "qtea_rows_plan_shapes")
    return dict(grid=plan[0], rows_cap=plan[1], wide=plan[2], kparts=plan[3], ctas=[ctas[i] for i in range(n)])


def qtea_device_status(layout: Layout, stream=None) -> int:
    return load().qtea_device_status(layout.handle, _stream(stream))


def qtea_probe_decode_rates() -> dict:
    """Cycles per instruction per SM sub-partition of the instructions a batch-1 decode could run
    on (a diagnostic behind the dp4a decode; see include/qtea.h)."""
    out = (ctypes.c_double * 5)()
    rc = load().qtea_probe_decode_rates(out, 5)
    if rc:
        raise QteaError(rc, "qtea_probe_decode_rates")
    names = ("mma_m16n8k16_f16_constant", "mma_m16n8k16_f16_decoded_a", "mma_m16n8k32_e4m3_constant",
             "mma_m16n8k32_e4m3_decoded_a", "dp4a")
    return {n: round(out[i], 3) for i, n in enumerate(names)}


def packed_bytes(layout: Layout):
    """Copy of the packed ternary bytes as a CUDA uint8 tensor (for inspection and tests)."""
    import torch
    n = layout.describe()["packed_bytes"]
    out = torch.empty(max(n, 1), dtype=torch.uint8, device="cuda")
    rc = load().qtea_layout_copy_packed(layout.handle, out.data_ptr(), n, _stream(None))
    if rc:
        raise QteaError(rc, "qtea_layout_copy_packed")
    return out[:n]


def qtea_quantize(W, hdiag, group_size: Optional[int] = None, n_salient: int = 0, bias: bool = False,
                  fit_iters: int = 4, rescale_iters: int = 2, stream=None) -> dict:
    """The quantizer's per-layer steps on the GPU: fp32 weights W [N][K] and diag(H) [K] (CUDA
    tensors) to the GEMV's inputs. Returns a dict of CUDA tensors: codes int8 [N][K], row_scale
    int16 (fp16 bits) [N][G] or [N][2G] with bias, col_scale [K], salient_idx int32 [s],
    residual_vals [N/4][s] and residual_idx uint8 [N/4][ceil(s/4)]."""
    import torch
    if W.dim() != 2:
        raise ValueError("W must be [N][K]")
    N, K = W.shape
    g = K if group_size is None else int(group_size)
    G = (K + g - 1) // g if g > 0 else 1
    s = int(n_salient)
    dev = W.device
    out = dict(
        codes=torch.empty((N, K), dtype=torch.int8, device=dev),
        row_scale=torch.empty((N, G * (2 if bias else 1)), dtype=torch.int16, device=dev),
        col_scale=torch.empty((K,), dtype=torch.int16, device=dev),
        salient_idx=torch.empty((s,), dtype=torch.int32, device=dev),
        residual_vals=torch.empty((N // 4, s), dtype=torch.int16, device=dev),
        residual_idx=torch.empty((N // 4, (s + 3) // 4), dtype=torch.uint8, device=dev),
    )
    rc = load().qtea_quantize(
        _ptr(W, (torch.float32,), "W"), _ptr(hdiag, (torch.float32,), "hdiag", (K,)), N, K, g, s,
        QTEA_OPT_BIAS if bias else 0, int(fit_iters), int(rescale_iters), out["codes"].data_ptr(),
        out["row_scale"].data_ptr(), out["col_scale"].data_ptr(), out["salient_idx"].data_ptr() if s else None,
        out["residual_vals"].data_ptr() if s else None, out["residual_idx"].data_ptr() if s else None,
        _stream(stream))
    if rc:
        raise QteaError(rc, "qtea_quantize")
    return out


def qtea_salient_from_bitmap(bitmap, K: int, max_s: Optional[int] = None, stream=None):
    """Sec. 3.5's salient bitmap (int32 or uint32 CUDA tensor of ceil(K/32) words, column j at bit
    j % 32 of word j // 32) as the ascending int32 index list qtea_gemv takes."""
    import torch
    words = (K + 31) // 32
    ptr = _ptr(bitmap, (torch.int32,) + ((torch.uint32,) if hasattr(torch, "uint32") else ()), "bitmap", (words,))
    max_s = K if max_s is None else int(max_s)
    out = torch.empty(max(max_s, 1), dtype=torch.int32, device=bitmap.device)
    n = ctypes.c_int32(0)
    rc = load().qtea_salient_from_bitmap(ptr, int(K), out.data_ptr(), max_s, ctypes.byref(n), _stream(stream))
    if rc != QTEA_OK:
        raise QteaError(rc, "qtea_salient_from_bitmap")
    return out[:n.value]


def qtea_salient_to_bitmap(salient_idx, K: int, stream=None):
    """The bitmap (int32 CUDA tensor of ceil(K/32) words holding the uint32 bits) of a strictly
    ascending int32 salient index list."""
    import torch
    s = 0 if salient_idx is None else int(salient_idx.numel())
    ptr = _ptr(salient_idx, (torch.int32,), "salient_idx") if s else None
    dev = salient_idx.device if salient_idx is not None else torch.device("cuda")
    out = torch.empty(max((K + 31) // 32, 1), dtype=torch.int32, device=dev)
    rc = load().qtea_salient_to_bitmap(ptr, s, int(K), out.data_ptr(), _stream(stream))
    if rc != QTEA_OK:
        raise QteaError(rc, "qtea_salient_to_bitmap")
    return out[:(K + 31) // 32]
