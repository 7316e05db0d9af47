"""GPU parity for the quantizer's per-layer steps (Sec. 3.1-3.3, the 1:4 residual of Sec. 3.2 / 3.5):
every output of qtea_quantize bit-identical to the oracle's float32 steps (codes, binary16 alpha,
beta and v, salient columns, residual values and positions), and the quantized layer fed straight
into the GEMV.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle import quantize as oq

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qt():
    import paper_2609_00224_gb300 as m
    m.load()
    return m


def run(qt, W, h, group, s, bias, fit_iters=4, rescale_iters=2):
    out = qt.qtea_quantize(torch.from_numpy(W).cuda(), torch.from_numpy(h).cuda(), group_size=group, n_salient=s,
                           bias=bias, fit_iters=fit_iters, rescale_iters=rescale_iters)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def assert_same(got, ref, s):
    assert np.array_equal(got["salient_idx"], ref["salient_idx"]), "salient columns"
    assert np.array_equal(got["codes"], ref["codes"]), f"codes: {(got['codes'] != ref['codes']).sum()} differ"
    assert np.array_equal(got["row_scale"].view(np.uint16), ref["row_scale"]), "row_scale"
    assert np.array_equal(got["col_scale"].view(np.uint16), ref["col_scale"]), "col_scale"
    if s:
        assert np.array_equal(got["residual_vals"].view(np.uint16), ref["residual_vals"]), "residual values"
        assert np.array_equal(got["residual_idx"], ref["residual_idx"]), "residual positions"


CASES = [
    # N, K, group (None = K), s, bias
    (64, 300, 128, 16, True),   # ragged last group, s a multiple of 4
    (64, 300, 128, 16, False),
    (36, 256, None, 5, False),  # one alpha per row, s ragged against the position bytes
    (128, 1024, 128, 33, True),
    (8, 7, None, 3, True),      # K below one group
    (4, 1, None, 1, False),     # one column
    (16, 40, None, 40, True),   # every column salient
    (12, 513, 128, 0, True),    # no salient columns
    (32, 5000, 128, 520, False),  # the compaction's segments several columns long
    (20, 272, 128, 8, True),    # K % 32 == 16: the last 32-column block ends past the row (streamed sums)
    (36, 144, None, 8, False),  # the same with one group per row
    (300, 1056, 128, 12, True),  # 128-row tiles with a ragged last tile
    (6, 50, None, 0, True),     # no residual: N need not be a multiple of 4
]


@pytest.mark.parametrize("N,K,group,s,bias", CASES)
def test_quantize_is_bit_identical_to_oracle(qt, N, K, group, s, bias):
    W, h = synth.quant_problem(N * 7 + K + s, N, K)
    g = group or K
    assert_same(run(qt, W, h, g, s, bias), oq.quantize(W, h, g, s, bias), s)


@pytest.mark.parametrize("fit_iters,rescale_iters", [(0, 0), (0, 3), (7, 0), (1, 1)])
def test_iteration_counts(qt, fit_iters, rescale_iters):
    W, h = synth.quant_problem(3, 48, 384)
    got = run(qt, W, h, 128, 12, True, fit_iters, rescale_iters)
    assert_same(got, oq.quantize(W, h, 128, 12, True, fit_iters, rescale_iters), 12)
    if rescale_iters == 0:
        assert np.all(got["col_scale"].view(np.uint16) == 0x3C00)  # v = 1


def test_ties(qt):
    """Coarse weight values and a flat h: many equal salient scores (lower column wins) and equal
    |r| inside groups of four rows (lower row wins), plus all-zero groups (alpha = 0, T = 0)."""
    rng = np.random.default_rng(11)
    N, K = 32, 256
    W = (rng.integers(-3, 4, size=(N, K)) * 0.125).astype(np.float32)
    W[4:8] = W[0:4]          # identical rows inside one group of four
    W[8:12, :] = W[8, :]     # four equal rows
    W[:, 128:] *= (np.arange(K - 128) % 2 == 0)[None, :]
    W[16, :128] = 0.0        # an all-zero group
    h = np.ones(K, np.float32)
    for bias in (False, True):
        assert_same(run(qt, W, h, 128, 40, bias), oq.quantize(W, h, 128, 40, bias), 40)


def test_llama_shape_sample(qt):
    """A full-width row block of a Llama3-8B q_proj shape (K = 4096) with the paper's salient count
    scale (1 % of K): several hundred rows, every column."""
    W, h = synth.quant_problem(21, 256, 4096)
    assert_same(run(qt, W, h, 128, 41, True), oq.quantize(W, h, 128, 41, True), 41)


def test_down_proj_width(qt):
    """The widest Llama3-8B input (K = 14336, down_proj) on a 1024-row slice: 448 column blocks in
    the streamed column sums, 112 groups per row, 8 row tiles, the GEMV's salient count."""
    W, h = synth.quant_problem(33, 1024, 14336)
    assert_same(run(qt, W, h, 128, 432, True), oq.quantize(W, h, 128, 432, True), 432)


@pytest.mark.parametrize("bias", [False, True])
def test_quantized_layer_through_the_gemv(qt, bias):
    """qtea_quantize's outputs go straight into qtea_pack_layout + qtea_gemv; the result matches the
    oracle GEMV on the oracle quantizer's outputs (which are the same bits)."""
    N, K, s, g = 256, 1024, 24, 128
    W, h = synth.quant_problem(5, N, K)
    out = qt.qtea_quantize(torch.from_numpy(W).cuda(), torch.from_numpy(h).cuda(), group_size=g, n_salient=s,
                           bias=bias)
    layout = qt.qtea_pack_layout(out["codes"], n_salient=s, group_size=g)
    if bias:
        layout.set_options(qt.QTEA_OPT_BIAS)
    xs = synth.normal_f16(9, 42, (4, K), 0.0, 0.5)
    x = torch.from_numpy(xs.view(np.int16)).cuda().view(torch.float16)
    f16 = lambda t: t.view(torch.float16)
    y = qt.qtea_gemv(x, layout, f16(out["row_scale"]), f16(out["col_scale"]), out["salient_idx"],
                     f16(out["residual_vals"]), out["residual_idx"])
    torch.cuda.synchronize()
    ref = oq.quantize(W, h, g, s, bias)
    y_ref, bound = oracle.gemv(xs, ref["codes"], ref["alpha"].reshape(N, -1), ref["col_scale"], ref["salient_idx"],
                               ref["residual_vals"], ref["residual_idx"],
                               beta=ref["beta"].reshape(N, -1) if bias else None, group_size=g)
    err = np.abs(y.cpu().numpy().astype(np.float64) - y_ref)
    assert np.all(err <= 1e-4 * bound + 1e-6)
