"""QTEA quantizer steps, plain and slow (test infrastructure: only tests/, __graft_entry__.smoke()
and bench.py's CPU baseline use it).

The per-layer steps of the method, without the GPTQ-style error propagation of Sec. 3.4:
  * salient-column scores s_j = max_i W_ij^2 * diag(H)_j^2 and the top-s selection (Sec. 3.2);
  * ternary assignment T = nearest point of {beta - alpha, beta, beta + alpha} (Sec. 3.1, Eq. 2-3),
    alpha and beta per row and group;
  * column-wise rescale refinement v_j = mean_{i: T_ij != 0} |W_ij - beta_i| / alpha_i, alternated
    with reassignment to {beta - v_j alpha, beta, beta + v_j alpha} (Sec. 3.3, Eq. 6-7);
  * the 1:4 residual on the salient columns (Sec. 3.2, Sec. 3.5): per group of four rows the entry
    with the largest |W - W^| and its value.

Readings (the paper is silent on these; see the design notes): beta is the group mean (zero
without the bias option), alpha starts at the group's mean |W - beta| and is refitted as the mean
|W - beta| over the nonzero codes for `fit_iters` rounds (the least-squares alpha for fixed T);
ties in the salient ranking go to the lower column, ties of |r| to the lower row. Decisions that
produce integers (codes, salient columns, positions) are taken in float32 with every sum formed in
a fixed sequential order, which the GPU kernels reproduce exactly; alpha, beta and v are stored as
binary16 (round to nearest even), and the residual is measured against the stored values.
"""
from __future__ import annotations

import numpy as np

F = np.float32


def _seq_sum(a: np.ndarray, axis: int) -> np.ndarray:
    """Sum in index order along `axis`, in float32 (one rounding per addition)."""
    a = np.moveaxis(np.asarray(a, F), axis, 0)
    acc = np.zeros(a.shape[1:], F)
    for k in range(a.shape[0]):
        acc = (acc + a[k]).astype(F)
    return acc


def salient_scores(W: np.ndarray, h: np.ndarray) -> np.ndarray:
    """Sec. 3.2: s_j = max_i W_ij^2 * diag(H)_j^2 (float32; the max of the rounded squares, times
    the rounded h_j^2)."""
    w2 = (W.astype(F) * W.astype(F)).astype(F)
    hh = (h.astype(F) * h.astype(F)).astype(F)
    return (w2.max(axis=0) * hh).astype(F)


def select_salient(score: np.ndarray, s: int) -> np.ndarray:
    """The s highest scores (ties: lower column first), returned in ascending column order."""
    K = score.shape[0]
    order = np.lexsort((np.arange(K), -score.astype(np.float64)))
    return np.sort(order[:s]).astype(np.int32)


def _assign(d: np.ndarray, half: np.ndarray) -> np.ndarray:
    """Nearest point of {-a, 0, +a} for d with threshold half = a / 2 (Eq. 3)."""
    return np.where(d > half, 1, np.where(d < -half, -1, 0)).astype(np.int8)


def group_fit(W: np.ndarray, group: int, bias: bool, fit_iters: int):
    """Sec. 3.1: per row and group of `group` columns, beta (the group mean, or 0), alpha (mean
    |W - beta|, then refitted over the nonzero codes `fit_iters` times) and the ternary codes.
    Returns alpha, beta [N][G] float32 and T [N][K] int8."""
    N, K = W.shape
    G = -(-K // group)
    alpha = np.zeros((N, G), F)
    beta = np.zeros((N, G), F)
    T = np.zeros((N, K), np.int8)
    for gi in range(G):
        cols = W[:, gi * group:min(K, (gi + 1) * group)].astype(F)
        n = F(cols.shape[1])
        b = (_seq_sum(cols, 1) / n).astype(F) if bias else np.zeros(N, F)
        d = (cols - b[:, None]).astype(F)
        ad = np.abs(d)
        a = (_seq_sum(ad, 1) / n).astype(F)
        for _ in range(fit_iters):
            t = _assign(d, (a * F(0.5)).astype(F)[:, None])
            num = _seq_sum(np.where(t != 0, ad, F(0)), 1)
            cnt = (t != 0).sum(axis=1)
            with np.errstate(divide="ignore", invalid="ignore"):  # all-zero groups keep alpha
                a = np.where(cnt > 0, (num / cnt.astype(F)).astype(F), a).astype(F)
        T[:, gi * group:gi * group + cols.shape[1]] = _assign(d, (a * F(0.5)).astype(F)[:, None])
        alpha[:, gi] = a
        beta[:, gi] = b
    return alpha, beta, T


def column_rescale(W: np.ndarray, alpha: np.ndarray, beta: np.ndarray, T: np.ndarray, group: int,
                   iters: int):
    """Sec. 3.3, Eq. 6-7: `iters` rounds of v_j = mean over rows with T_ij != 0 of
    |W_ij - beta_i| / alpha_i (rows in order; v_j = 1 when no code of the column is nonzero), then
    reassignment to the nearest of {beta - v_j alpha, beta, beta + v_j alpha}. Returns v [K] float32
    and the final T."""
    N, K = W.shape
    gidx = np.arange(K) // group
    a = alpha[:, gidx].astype(F)
    b = beta[:, gidx].astype(F)
    d = (W.astype(F) - b).astype(F)
    ad = np.abs(d)
    v = np.ones(K, F)
    T = T.copy()
    with np.errstate(divide="ignore", invalid="ignore"):
        term = (ad / a).astype(F)
    for _ in range(iters):
        acc = np.zeros(K, F)
        cnt = np.zeros(K, np.int64)
        for i in range(N):
            nz = T[i] != 0
            acc = np.where(nz, (acc + term[i]).astype(F), acc).astype(F)
            cnt += nz
        with np.errstate(divide="ignore", invalid="ignore"):  # columns without nonzero codes keep v
            v = np.where(cnt > 0, (acc / cnt.astype(F)).astype(F), v).astype(F)
        half = ((v[None, :] * a).astype(F) * F(0.5)).astype(F)
        T = _assign(d, half)
    return v, T


def _f16(x: np.ndarray) -> np.ndarray:
    return np.asarray(x, F).astype(np.float16)


def residual_1of4(W: np.ndarray, T: np.ndarray, alpha16: np.ndarray, beta16: np.ndarray, v16: np.ndarray,
                  salient: np.ndarray, group: int):
    """Sec. 3.2 / 3.5: on every salient column j and group of four rows, the row whose
    r = W - (alpha v T + beta) (float32, from the stored binary16 alpha, beta, v) has the largest
    |r| (ties: lower row), its position and r rounded to binary16. Returns values [N/4][s] (fp16
    bits) and packed positions [N/4][ceil(s/4)] (entry c at bits 2(c % 4) of byte c / 4)."""
    N, K = W.shape
    s = salient.shape[0]
    vals = np.zeros((N // 4, s), np.uint16)
    ridx = np.zeros((N // 4, (s + 3) // 4), np.uint8)
    for c, j in enumerate(salient):
        gi = j // group
        a = alpha16[:, gi].astype(F)
        b = beta16[:, gi].astype(F)
        what = ((a * F(v16[j])).astype(F) * T[:, j].astype(F)).astype(F)
        what = (what + b).astype(F)
        r = (W[:, j].astype(F) - what).astype(F).reshape(N // 4, 4)
        pos = np.argmax(np.abs(r), axis=1)
        vals[:, c] = _f16(r[np.arange(N // 4), pos]).view(np.uint16)
        ridx[:, c // 4] |= (pos.astype(np.uint8) << np.uint8(2 * (c % 4)))
    return vals, ridx


def quantize(W: np.ndarray, h: np.ndarray, group: int, s: int, bias: bool, fit_iters: int = 4,
             rescale_iters: int = 2) -> dict:
    """All steps in the paper's order: scores and salient columns, group fit, column rescale,
    binary16 rounding, residual. The outputs are the GEMV's inputs: codes, row_scale (alpha, or
    (alpha, beta) pairs with bias), col_scale v, salient list, residual values and positions."""
    N, K = W.shape
    sal = select_salient(salient_scores(W, h), s)
    alpha, beta, T = group_fit(W, group, bias, fit_iters)
    v, T = column_rescale(W, alpha, beta, T, group, rescale_iters)
    alpha16, beta16, v16 = _f16(alpha), _f16(beta), _f16(v)
    vals, ridx = residual_1of4(W, T, alpha16, beta16, v16, sal, group)
    if bias:
        row_scale = np.stack([alpha16, beta16], axis=-1).reshape(N, -1)
    else:
        row_scale = alpha16
    return dict(codes=T, alpha=alpha16.view(np.uint16), beta=beta16.view(np.uint16),
                row_scale=np.ascontiguousarray(row_scale).view(np.uint16), col_scale=v16.view(np.uint16),
                salient_idx=sal, residual_vals=vals, residual_idx=ridx, alpha32=alpha, beta32=beta, v32=v)
