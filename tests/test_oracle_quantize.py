"""Pins of the oracle quantizer (oracle/quantize.py) against what the paper's definitions fix:
a hand-worked example (tests/golden/quant_example.txt), the nearest-point property of the codes
(Sec. 3.1 Eq. 3), the fixed points of alpha and v (the means they are defined as, Sec. 3.1 and
Sec. 3.3 Eq. 7), the salient ranking (Sec. 3.2) and the 1:4 residual (largest |W - W^| per group of
four), all recomputed independently in float64; the output formats are pinned by running the GEMV
oracle on them. Mutants of the quantizer's source must each fail a pin."""
import os
import types

import numpy as np
import pytest

import oracle
import synth
from oracle import quantize as Q

HERE = os.path.dirname(os.path.abspath(__file__))


def golden():
    vals = {}
    for line in open(os.path.join(HERE, "golden", "quant_example.txt")):
        if line.startswith("#") or not line.strip():
            continue
        k, *rest = line.split()
        vals[k] = [float(t) for t in rest]
    return vals


def run_example(mod):
    g = golden()
    W = np.array(g["W"], np.float32).reshape(4, 4)
    h = np.ones(4, np.float32)
    return g, mod.quantize(W, h, 4, 1, True, fit_iters=2, rescale_iters=1)


def check_example(mod):
    g, out = run_example(mod)
    assert out["codes"].reshape(-1).tolist() == [int(t) for t in g["codes"]]
    assert np.allclose(out["alpha32"][:, 0], g["alpha"], rtol=1e-6, atol=1e-7)
    assert np.allclose(out["beta32"][:, 0], g["beta"], rtol=1e-6, atol=1e-7)
    assert np.allclose(out["v32"], g["v"], rtol=1e-6)
    assert out["salient_idx"].tolist() == [int(t) for t in g["salient"]]
    pos = int(out["residual_idx"][0, 0] & 3)
    assert pos == int(g["residual_position"][0])
    val = float(out["residual_vals"][0, 0:1].view(np.float16)[0])
    assert abs(val - g["residual_value"][0]) < 2e-4


def check_properties(mod, N=64, K=300, group=128, s=16, bias=True, seed=3):
    W, h = synth.quant_problem(seed, N, K)
    out = mod.quantize(W, h, group, s, bias, fit_iters=3, rescale_iters=1)
    W64 = W.astype(np.float64)
    G = -(-K // group)
    gidx = np.arange(K) // group
    # group fit alone: beta is the group mean, alpha the mean |d| over the nonzero codes, and the
    # codes are the nearest points for that alpha
    a32, b32, T0 = mod.group_fit(W, group, bias, 3)
    for gi in range(G):
        cols = W64[:, gi * group:min(K, (gi + 1) * group)]
        b = cols.mean(axis=1) if bias else np.zeros(N)
        assert np.allclose(b32[:, gi], b, rtol=1e-5, atol=1e-7)
        d = cols - b32[:, gi:gi + 1]
        t = T0[:, gi * group:gi * group + cols.shape[1]]
        near = np.where(d > a32[:, gi:gi + 1] / 2, 1, np.where(d < -a32[:, gi:gi + 1] / 2, -1, 0))
        assert (near == t).mean() > 0.999
    # v: the mean |W - beta| / alpha over the nonzero group-fit codes of the column
    d_all = W64 - b32[:, gidx]
    with np.errstate(divide="ignore", invalid="ignore"):
        ratio = np.abs(d_all) / a32[:, gidx]
    nz = T0 != 0
    v_ref = np.where(nz.sum(0) > 0, np.where(nz, ratio, 0).sum(0) / np.maximum(nz.sum(0), 1), 1.0)
    assert np.allclose(out["v32"], v_ref, rtol=1e-5)
    # final codes: nearest points for v_j alpha_i
    half = out["v32"][None, :].astype(np.float64) * a32[:, gidx] / 2
    near = np.where(d_all > half, 1, np.where(d_all < -half, -1, 0))
    assert (near == out["codes"]).mean() > 0.999
    # salient columns: the s largest max_i W_ij^2 h_j^2
    score = (W64 ** 2).max(axis=0) * h.astype(np.float64) ** 2
    top = np.sort(np.argsort(-score, kind="stable")[:s])
    assert out["salient_idx"].tolist() == top.tolist()
    # residual: the largest |W - W^| of each group of four on each salient column
    a16 = out["alpha"].view(np.float16).astype(np.float64)
    b16 = out["beta"].view(np.float16).astype(np.float64)
    v16 = out["col_scale"].view(np.float16).astype(np.float64)
    pos = synth.residual_positions(out["residual_idx"], s)
    vals = out["residual_vals"].view(np.float16).astype(np.float64)
    for c, j in enumerate(out["salient_idx"]):
        what = a16[:, j // group] * v16[j] * out["codes"][:, j] + b16[:, j // group]
        r = (W64[:, j] - what).reshape(N // 4, 4)
        assert (np.argmax(np.abs(r), axis=1) == pos[:, c]).mean() > 0.99
        rsel = r[np.arange(N // 4), pos[:, c]]
        assert np.allclose(vals[:, c], rsel, rtol=1e-3, atol=1e-7)
    return W, h, out


def test_worked_example():
    check_example(Q)


@pytest.mark.parametrize("bias", [True, False])
@pytest.mark.parametrize("N,K,group,s", [(64, 300, 128, 16), (32, 256, 256, 8), (128, 1024, 128, 24)])
def test_definitions_hold(N, K, group, s, bias):
    check_properties(Q, N, K, group, s, bias)


def test_codes_are_ternary_and_formats_feed_the_gemv():
    W, h, out = check_properties(Q, 64, 512, 128, 16, True, seed=9)
    assert set(np.unique(out["codes"])) <= {-1, 0, 1}
    # the quantized layer through the GEMV oracle equals the dense dequantized product
    x = synth.normal_f16(5, 1, (2, 512), 0.0, 1.0)
    y, _ = oracle.gemv(x, out["codes"], out["alpha"], out["col_scale"], out["salient_idx"], out["residual_vals"],
                       out["residual_idx"], beta=out["beta"], group_size=128)
    a16 = out["alpha"].view(np.float16).astype(np.float64)
    b16 = out["beta"].view(np.float16).astype(np.float64)
    v16 = out["col_scale"].view(np.float16).astype(np.float64)
    g = np.arange(512) // 128
    Wh = a16[:, g] * v16[None, :] * out["codes"] + b16[:, g]
    pos = synth.residual_positions(out["residual_idx"], 16)
    vals = out["residual_vals"].view(np.float16).astype(np.float64)
    for c, j in enumerate(out["salient_idx"]):
        Wh[np.arange(16) * 4 + pos[:, c], j] += vals[:, c]
    assert np.allclose(y, x.view(np.float16).astype(np.float64) @ Wh.T, rtol=1e-9, atol=1e-9)
    # and the quantization error is what the residual leaves: the residual removes the largest
    # error of every group of four on the salient columns
    assert np.abs(W.astype(np.float64) - Wh)[:, out["salient_idx"]].max() <= \
        np.abs(W.astype(np.float64) - (a16[:, g] * v16[None, :] * out["codes"] + b16[:, g]))[:, out["salient_idx"]].max()


MUTANTS = {
    "beta_not_mean": ("(_seq_sum(cols, 1) / n).astype(F) if bias", "(_seq_sum(cols, 1) / (n + 1)).astype(F) if bias"),
    "threshold_alpha": ("return np.where(d > half, 1, np.where(d < -half, -1, 0))",
                        "return np.where(d > 2 * half, 1, np.where(d < -2 * half, -1, 0))"),
    "alpha_max": ("num = _seq_sum(np.where(t != 0, ad, F(0)), 1)",
                  "num = np.where(t != 0, ad, F(0)).max(1) * (t != 0).sum(axis=1)"),
    "v_no_alpha": ("term = (ad / a).astype(F)", "term = (ad / F(1)).astype(F)"),
    "score_no_h": ("return (w2.max(axis=0) * hh).astype(F)", "return w2.max(axis=0)"),
    "residual_argmin": ("pos = np.argmax(np.abs(r), axis=1)", "pos = np.argmin(np.abs(r), axis=1)"),
    "residual_no_beta": ("what = (what + b).astype(F)", "what = what"),
    "salient_lowest": ("order = np.lexsort((np.arange(K), -score.astype(np.float64)))",
                       "order = np.lexsort((np.arange(K), score.astype(np.float64)))"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutants_fail_a_pin(name):
    old, new = MUTANTS[name]
    src = open(Q.__file__).read()
    assert src.count(old) == 1, name
    mod = types.ModuleType("quantize_mutant")
    exec(compile(src.replace(old, new), "quantize_mutant", "exec"), mod.__dict__)
    failed = False
    for check in (lambda: check_example(mod), lambda: check_properties(mod), lambda: check_properties(mod, bias=False)):
        try:
            check()
        except AssertionError:
            failed = True
    assert failed, f"mutant {name} passed every pin"
