"""Python access to the QTEA oracle (``qtea_oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` use this module; the GPU library and its binding never import it.
This file only marshals numpy arrays into the C routines; all arithmetic is in the C
file, which follows Eq. 4, Eq. 10 and Eq. 11 of the QTEA paper (Sec. 3.3 and 3.5).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qtea_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libqtea_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C, -O2, no fast-math) if it is missing or stale."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def load(path: str | None = None):
    """Load the oracle library (building it first); ``path`` selects another build of it."""
    global _lib
    if path is None and _lib is not None:
        return _lib
    lib = ctypes.CDLL(path or build())
    P = ctypes.c_void_p
    i32 = ctypes.c_int
    lib.qo_half_to_double.restype = ctypes.c_double
    lib.qo_half_to_double.argtypes = [ctypes.c_uint16]
    lib.qo_e4m3_to_double.restype = ctypes.c_double
    lib.qo_e4m3_to_double.argtypes = [ctypes.c_uint8]
    lib.qo_gemv.restype = i32
    lib.qo_gemv.argtypes = [i32, i32, i32, i32, P, P, P, P, P, i32, P, P, P, P, i32, P, P]
    lib.qo_gemv_ex.restype = i32
    lib.qo_gemv_ex.argtypes = [i32, i32, i32, i32, P, P, P, P, P, i32, P, P, i32, P, P, i32, P, P]
    for name in ("qo_pack_2bit", "qo_unpack_2bit", "qo_pack_base3", "qo_unpack_base3"):
        getattr(lib, name).restype = i32
        getattr(lib, name).argtypes = [P, i32, i32, P]
    lib.qo_packed_bytes_2bit.restype = ctypes.c_size_t
    lib.qo_packed_bytes_2bit.argtypes = [i32, i32]
    lib.qo_packed_bytes_base3.restype = ctypes.c_size_t
    lib.qo_packed_bytes_base3.argtypes = [i32, i32]
    lib.qo_lut5.restype = None
    lib.qo_lut5.argtypes = [P, P]
    lib.qo_salient_from_bitmap.restype = i32
    lib.qo_salient_from_bitmap.argtypes = [P, i32, P, i32]
    lib.qo_salient_to_bitmap.restype = i32
    lib.qo_salient_to_bitmap.argtypes = [P, i32, i32, P]
    lib.qo_asic_latency_us.restype = None
    lib.qo_asic_latency_us.argtypes = [i32, i32, P, P]
    if path is None:
        _lib = lib
    return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    pass


def half_to_double(h: int, lib=None) -> float:
    return (lib or load()).qo_half_to_double(int(h) & 0xFFFF)


def e4m3_to_double(b: int, lib=None) -> float:
    return (lib or load()).qo_e4m3_to_double(int(b) & 0xFF)


def gemv(x, T, alpha, v, salient_idx=None, residual_vals=None, residual_idx=None, beta=None,
         group_size=None, rows=None, want_bound=True, residual_fp8=False, lib=None):
    """y = x * W^T per Eq. 10/11 in fp64. fp16 inputs are given as uint16 bit patterns.

    x [M][K] uint16, T [N][K] int8, alpha [N][G] uint16, v [K] uint16, beta [N][G] uint16 or None,
    salient_idx [s] int32, residual_vals [N/4][s] uint16 (uint8 FP8 E4M3 bytes with
    residual_fp8), residual_idx [N/4][ceil(s/4)] uint8.
    Returns (y, bound), each float64 [M][n_out].
    """
    lib = lib or load()
    x = _c(np.atleast_2d(x), np.uint16)
    T = _c(T, np.int8)
    M, K = x.shape
    N = T.shape[0]
    if T.shape[1] != K:
        raise ValueError("x and T disagree on K")
    group_size = K if group_size is None else int(group_size)
    if group_size <= 0:
        group_size = max(K, 1)
    s = 0 if salient_idx is None else int(np.asarray(salient_idx).size)
    rows_a = None if rows is None else _c(rows, np.int32)
    n_out = N if rows_a is None else rows_a.size
    y = np.zeros((M, n_out), np.float64)
    b = np.zeros((M, n_out), np.float64) if want_bound else None
    alpha = _c(alpha, np.uint16)
    beta = _c(beta, np.uint16)
    v = _c(v, np.uint16)
    si = _c(salient_idx, np.int32) if s else None
    rv = _c(residual_vals, np.uint8 if residual_fp8 else np.uint16) if s else None
    ri = _c(residual_idx, np.uint8) if s else None
    rc = lib.qo_gemv_ex(M, N, K, group_size, _ptr(T), _ptr(x), _ptr(alpha), _ptr(beta), _ptr(v), s,
                        _ptr(si), _ptr(rv), int(bool(residual_fp8)), _ptr(ri), _ptr(rows_a), n_out, _ptr(y),
                        _ptr(b))
    if rc != 0:
        raise OracleError(f"qo_gemv returned {rc}")
    return y, b


def packed_bytes(N: int, K: int, fmt: str = "2bit", lib=None) -> int:
    lib = lib or load()
    return int(lib.qo_packed_bytes_2bit(N, K) if fmt == "2bit" else lib.qo_packed_bytes_base3(N, K))


def pack(T, fmt: str = "2bit", lib=None) -> np.ndarray:
    lib = lib or load()
    T = _c(T, np.int8)
    N, K = T.shape
    out = np.zeros(packed_bytes(N, K, fmt, lib), np.uint8)
    fn = lib.qo_pack_2bit if fmt == "2bit" else lib.qo_pack_base3
    rc = fn(_ptr(T), N, K, _ptr(out))
    if rc != 0:
        raise OracleError(f"pack returned {rc}")
    return out


def unpack(packed, N: int, K: int, fmt: str = "2bit", lib=None) -> np.ndarray:
    lib = lib or load()
    packed = _c(packed, np.uint8)
    if packed.size != packed_bytes(N, K, fmt, lib):
        raise ValueError("packed size does not match N, K")
    T = np.zeros((N, K), np.int8)
    fn = lib.qo_unpack_2bit if fmt == "2bit" else lib.qo_unpack_base3
    rc = fn(_ptr(packed), N, K, _ptr(T))
    if rc != 0:
        raise OracleError(f"unpack returned {rc}")
    return T


def salient_from_bitmap(bitmap, K: int, lib=None) -> np.ndarray:
    """Sec. 3.5's salient bitmap (uint32 words, column j at bit j % 32 of word j // 32) as the
    ascending index list."""
    lib = lib or load()
    bitmap = _c(bitmap, np.uint32)
    if bitmap.size < (K + 31) // 32:
        raise ValueError("bitmap shorter than K bits")
    out = np.zeros(max(K, 1), np.int32)
    n = lib.qo_salient_from_bitmap(_ptr(bitmap), K, _ptr(out), K)
    if n < 0:
        raise OracleError(f"salient_from_bitmap returned {n}")
    return out[:n].copy()


def salient_to_bitmap(idx, K: int, lib=None) -> np.ndarray:
    """The bitmap of a strictly ascending salient index list (each in [0, K))."""
    lib = lib or load()
    idx = _c(idx, np.int32)
    out = np.zeros(max((K + 31) // 32, 1), np.uint32)
    rc = lib.qo_salient_to_bitmap(_ptr(idx), idx.size, K, _ptr(out))
    if rc != 0:
        raise OracleError(f"salient_to_bitmap returned {rc}")
    return out[:(K + 31) // 32].copy()


def lut5(xs, lib=None) -> np.ndarray:
    lib = lib or load()
    xs = _c(xs, np.float64)
    out = np.zeros(243, np.float64)
    lib.qo_lut5(_ptr(xs), _ptr(out))
    return out


def asic_latency_us(K: int, N: int, lib=None):
    lib = lib or load()
    a = np.zeros(1, np.float64)
    b = np.zeros(1, np.float64)
    lib.qo_asic_latency_us(int(K), int(N), _ptr(a), _ptr(b))
    return float(a[0]), float(b[0])
