"""Seeded synthetic inputs for the QTEA ternary + 1:4 residual GEMV.

This module draws the operands (ternary codes, per-row scale alpha, per-column rescale v,
activations x, salient columns, residual values and 1:4 positions) and rounds them to
their storage formats. It holds none of the GEMV arithmetic; the oracle and the GPU
library both consume exactly the bytes produced here.

The workload shapes stand in for real model weights (which are not available): the layer
shapes of Llama3-8B, Qwen3-14B and Llama3-70B, with random ternary codes and the value
distributions listed in ``WORKLOADS``.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
from typing import Dict, List, Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB_PATH = os.path.join(_HERE, "libqtea_synth.so")
_lib = None

# stream ids, one per tensor kind
S_CODES, S_ALPHA, S_V, S_X, S_SALIENT, S_RVALS, S_RIDX, S_BETA, S_MASSIVE = 1, 2, 3, 4, 5, 6, 7, 8, 9


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=gnu99", "-fPIC", "-shared", "-pthread", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    u64, sz, d, P, i32 = ctypes.c_uint64, ctypes.c_size_t, ctypes.c_double, ctypes.c_void_p, ctypes.c_int
    lib.synth_f16_from_double.restype = ctypes.c_uint16
    lib.synth_f16_from_double.argtypes = [d]
    lib.synth_codes.restype = None
    lib.synth_codes.argtypes = [u64, u64, sz, d, d, P]
    for n in ("synth_uniform_f16", "synth_normal_f16", "synth_laplace_f16"):
        getattr(lib, n).restype = None
        getattr(lib, n).argtypes = [u64, u64, sz, d, d, P]
    lib.synth_e4m3_from_double.restype = ctypes.c_uint8
    lib.synth_e4m3_from_double.argtypes = [d]
    lib.synth_normal_e4m3.restype = None
    lib.synth_normal_e4m3.argtypes = [u64, u64, sz, d, d, P]
    lib.synth_salient.restype = i32
    lib.synth_salient.argtypes = [u64, u64, i32, i32, P]
    lib.synth_residual_idx.restype = None
    lib.synth_residual_idx.argtypes = [u64, u64, i32, i32, P]
    _lib = lib
    return lib


def _p(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def f16_from_double(v: float) -> int:
    return int(_load().synth_f16_from_double(float(v)))


def codes(seed, stream, shape, p_neg, p_zero) -> np.ndarray:
    out = np.empty(shape, np.int8)
    _load().synth_codes(seed, stream, out.size, p_neg, p_zero, _p(out))
    return out


def e4m3_from_double(v: float) -> int:
    return int(_load().synth_e4m3_from_double(float(v)))


def normal_e4m3(seed, stream, shape, mean, std) -> np.ndarray:
    out = np.empty(shape, np.uint8)
    _load().synth_normal_e4m3(seed, stream, out.size, mean, std, _p(out))
    return out


def uniform_f16(seed, stream, shape, lo, hi) -> np.ndarray:
    out = np.empty(shape, np.uint16)
    _load().synth_uniform_f16(seed, stream, out.size, lo, hi, _p(out))
    return out


def normal_f16(seed, stream, shape, mean, std) -> np.ndarray:
    out = np.empty(shape, np.uint16)
    _load().synth_normal_f16(seed, stream, out.size, mean, std, _p(out))
    return out


def laplace_f16(seed, stream, shape, loc, scale) -> np.ndarray:
    out = np.empty(shape, np.uint16)
    _load().synth_laplace_f16(seed, stream, out.size, loc, scale, _p(out))
    return out


def salient(seed, stream, K, s) -> np.ndarray:
    out = np.empty(max(s, 0), np.int32)
    if _load().synth_salient(seed, stream, K, s, _p(out)) != 0:
        raise ValueError(f"cannot draw {s} salient columns out of {K}")
    return out


def residual_idx(seed, stream, n_groups, s) -> np.ndarray:
    out = np.empty((n_groups, (s + 3) // 4), np.uint8)
    _load().synth_residual_idx(seed, stream, n_groups, s, _p(out))
    return out


def residual_positions(ridx: np.ndarray, s: int) -> np.ndarray:
    """Unpacked view [n_groups][s] of the packed 2-bit positions (input-format helper)."""
    c = np.arange(s)
    return (ridx[:, c // 4] >> (2 * (c % 4)).astype(np.uint8)) & 3


def salient_count(K: int, frac: float = 0.03) -> int:
    """3% of the input columns, rounded half up to a multiple of 8."""
    return 8 * int(np.floor(frac * K / 8 + 0.5))


@dataclasses.dataclass
class Problem:
    name: str
    N: int
    K: int
    M: int
    s: int
    seed: int
    T: np.ndarray            # int8 [N][K]
    x: np.ndarray            # fp16 bits [M][K]
    alpha: np.ndarray        # fp16 bits [N][1]
    v: np.ndarray            # fp16 bits [K]
    salient_idx: np.ndarray  # int32 [s]
    residual_vals: np.ndarray  # fp16 bits [N/4][s] (uint8 FP8 E4M3 bytes when residual_fp8)
    residual_idx: np.ndarray   # uint8 [N/4][ceil(s/4)]
    group_size: int = 0        # columns per alpha (and beta) group; 0 = K (one per row)
    beta: Optional[np.ndarray] = None  # fp16 bits [N][G], or None (= 0)
    residual_fp8: bool = False

    @property
    def G(self) -> int:
        g = self.group_size or self.K
        return (self.K + g - 1) // g if self.K else 1


def make_problem(name: str, N: int, K: int, M: int, s: int, seed: int, p_neg: float = 0.3,
                 p_zero: float = 0.4, residual: str = "normal", residual_scale: float = 0.02,
                 alpha_range=(0.01, 0.05), v_range=(0.8, 1.2), group_size: int = 0, beta_std: float = 0.0,
                 residual_fp8: bool = False, x_std: float = 1.0) -> Problem:
    """Seeded operands (x drawn N(0, x_std)). group_size > 0 gives one alpha per (row, group of group_size columns),
    beta_std > 0 a per-(row, group) beta drawn N(0, beta_std), and residual_fp8 residual values
    rounded to FP8 E4M3 instead of fp16: the paper's own storage (Sec. 3.3, Eq. 4; Sec. 4.1)."""
    if s > 0 and N % 4:
        raise ValueError("N must be a multiple of 4 when there is a residual")
    g = group_size or K
    G = (K + g - 1) // g if K else 1
    T = codes(seed, S_CODES, (N, K), p_neg, p_zero)
    alpha = uniform_f16(seed, S_ALPHA, (N, G), *alpha_range)
    v = uniform_f16(seed, S_V, (K,), *v_range)
    x = normal_f16(seed, S_X, (M, K), 0.0, x_std)
    sal = salient(seed, S_SALIENT, K, s)
    if residual_fp8:
        if residual != "normal":
            raise ValueError("FP8 residual values are drawn from a normal distribution")
        rv = normal_e4m3(seed, S_RVALS, (N // 4, s), 0.0, residual_scale)
    elif residual == "normal":
        rv = normal_f16(seed, S_RVALS, (N // 4, s), 0.0, residual_scale)
    elif residual == "laplace":
        rv = laplace_f16(seed, S_RVALS, (N // 4, s), 0.0, residual_scale)
    elif residual == "zero":
        rv = np.zeros((N // 4, s), np.uint16)
    else:
        raise ValueError(residual)
    ri = residual_idx(seed, S_RIDX, N // 4, s)
    beta = normal_f16(seed, S_BETA, (N, G), 0.0, beta_std) if beta_std > 0 else None
    return Problem(name, N, K, M, s, seed, T, x, alpha, v, sal, rv, ri, group_size, beta, residual_fp8)


# Layer shapes (out x in) of the three model families the workloads are modelled on.
LLAMA3_8B = [("q_proj", 4096, 4096), ("k_proj", 1024, 4096), ("v_proj", 1024, 4096),
             ("o_proj", 4096, 4096), ("gate_proj", 14336, 4096), ("up_proj", 14336, 4096),
             ("down_proj", 4096, 14336)]
QWEN3_14B = [("q_proj", 5120, 5120), ("k_proj", 1024, 5120), ("v_proj", 1024, 5120),
             ("o_proj", 5120, 5120), ("gate_proj", 17408, 5120), ("up_proj", 17408, 5120),
             ("down_proj", 5120, 17408)]
LLAMA3_70B = [("q_proj", 8192, 8192), ("k_proj", 1024, 8192), ("v_proj", 1024, 8192),
              ("o_proj", 8192, 8192), ("gate_proj", 28672, 8192), ("up_proj", 28672, 8192),
              ("down_proj", 8192, 28672)]

# The workloads, by name. seed_base is the first seed of the workload: the operands of matrix j of
# layer l are drawn with seed seed_base + 16 l + j.
WORKLOADS: Dict[str, dict] = {
    "tiny_1024": dict(seed_base=0, shapes=[("tiny", 1024, 1024)], M=[1], p=(0.3, 0.4), residual="normal",
                      residual_scale=0.02, fixed_s=32),
    "llama3_8b_layer": dict(seed_base=1000, shapes=LLAMA3_8B, M=[1], p=(0.3, 0.4), residual="normal",
                            residual_scale=0.02),
    "qwen3_14b_layer": dict(seed_base=2000, shapes=QWEN3_14B, M=[1, 2, 4, 8, 16], p=(0.25, 0.5),
                            residual="normal", residual_scale=0.02),
    "llama3_70b_layer": dict(seed_base=3000, shapes=LLAMA3_70B, M=[1], p=(0.3, 0.4), residual="laplace",
                             residual_scale=0.01),
    "llama3_8b_32layer_stack": dict(seed_base=4000, shapes=LLAMA3_8B, M=[1], p=(0.3, 0.4), residual="normal",
                                    residual_scale=0.02, layers=32),
}


def workload_seed(workload: str, layer: int, matrix: int) -> int:
    return WORKLOADS[workload]["seed_base"] + 16 * layer + matrix


def workload_problem(workload: str, matrix: int, M: Optional[int] = None, layer: int = 0) -> Problem:
    cfg = WORKLOADS[workload]
    name, N, K = cfg["shapes"][matrix]
    s = cfg.get("fixed_s") or salient_count(K)
    M = cfg["M"][0] if M is None else M
    p_neg, p_zero = cfg["p"]
    return make_problem(f"{workload}/{name}", N, K, M, s, workload_seed(workload, layer, matrix), p_neg, p_zero,
                        cfg["residual"], cfg["residual_scale"])


# The paper's own storage of a layer (Sec. 3.3 and Sec. 4.1): alpha and beta per row and group of
# 128 columns, FP8 E4M3 residual values, base-3 codes. beta is drawn N(0, 0.002), a tenth of the
# typical |alpha * v| (the paper gives no distribution).
PAPER_FORMAT = dict(group_size=128, beta_std=0.002, residual_fp8=True)


def paper_problem(workload: str, matrix: int, M: Optional[int] = None, layer: int = 0,
                  residual_fp8: bool = True) -> Problem:
    """workload_problem's operands in the paper's storage (same seed, hence the same codes, x and
    v); residual_fp8=False keeps fp16 residual values with the paper's scale groups."""
    cfg = WORKLOADS[workload]
    name, N, K = cfg["shapes"][matrix]
    s = cfg.get("fixed_s") or salient_count(K)
    M = cfg["M"][0] if M is None else M
    p_neg, p_zero = cfg["p"]
    fmt = dict(PAPER_FORMAT, residual_fp8=residual_fp8)
    return make_problem(f"{workload}/{name}/paper_format", N, K, M, s, workload_seed(workload, layer, matrix), p_neg,
                        p_zero, "normal", cfg["residual_scale"], **fmt)


def plant_massive(x: np.ndarray, seed: int, magnitudes, lo: int = 0, hi: Optional[int] = None) -> np.ndarray:
    """Activations with a few "massive" values, as LLM hidden states show at some channels: a copy of
    x (fp16 bits [M][K]) in which len(magnitudes) distinct columns of [lo, hi), drawn with the seed,
    hold +-magnitude (alternating signs, every batch row), rounded to binary16. Returns the columns."""
    K = x.shape[-1]
    hi = K if hi is None else min(hi, K)
    n = len(magnitudes)
    cols = np.sort(salient(seed, S_MASSIVE, hi - lo, n) + lo)
    for i, (c, m) in enumerate(zip(cols, magnitudes)):
        x[..., c] = f16_from_double(float(m) if i % 2 == 0 else -float(m))
    return cols


def workload_shapes(workload: str) -> List[Tuple[str, int, int]]:
    return list(WORKLOADS[workload]["shapes"])


def quant_problem(seed: int, N: int, K: int, std: float = 0.02):
    """Inputs of the quantizer for one linear layer: full-precision weights W [N][K] (float32, drawn
    N(0, std) and rounded to binary16, so the same bytes feed every consumer) and a positive
    curvature diagonal h [K] standing in for diag(H) of a calibration set (float32,
    exp(N(0, 1)) rounded to binary16): the heavy-tailed spread that calibration Hessians show."""
    W = normal_f16(seed, 40, (N, K), 0.0, std).view(np.float16).astype(np.float32)
    z = normal_f16(seed, 41, (K,), 0.0, 1.0).view(np.float16).astype(np.float64)
    h = np.array([f16_from_double(float(np.exp(t))) for t in z], np.uint16).view(np.float16).astype(np.float32)
    return W, h
