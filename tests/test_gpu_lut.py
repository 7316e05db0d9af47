"""GPU parity of the table-lookup decode (the paper's Sec. 3.5 / Appendix A sign-symmetric LUT over
base-3 code bytes) against the fp64 oracle.

Pass rule (per output element): |y - y_ref| <= 1e-4 * sum_j |x_j * W^[o][j]| + 1e-6, the bound from
the oracle. The layouts are base-3 with one alpha per row (the table decode's default domain);
shapes cover several tiles and chunks, ragged K (a chunk shorter than 8 blocks, rows whose byte
length is not a multiple of 8), ragged N, no residual, every column salient, FP8 residual values and
massive activations.
"""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

REL, ABS = 1e-4, 1e-6


@pytest.fixture(scope="module")
def qt():
    import paper_2609_00224_gb300 as m
    m.load()
    return m


def dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.cuda()


def lut_layout(qt, p):
    layout = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, fmt=qt.QTEA_FMT_BASE3)
    layout.set_options(qt.QTEA_OPT_RESIDUAL_FP8 if p.residual_fp8 else 0)
    return layout


def args(p):
    f16 = lambda a: dev(np.ascontiguousarray(a).view(np.int16), torch.float16)
    rv = None
    if p.s:
        rv = dev(p.residual_vals) if p.residual_fp8 else f16(p.residual_vals)
    return dict(x=f16(p.x), row_scale=f16(p.alpha.reshape(-1)), col_scale=f16(p.v),
                salient_idx=dev(p.salient_idx) if p.s else None, residual_vals=rv,
                residual_idx=dev(p.residual_idx) if p.s else None)


def run(qt, p, layout=None):
    layout = layout or lut_layout(qt, p)
    a = args(p)
    y = qt.qtea_gemv(a["x"], layout, a["row_scale"], a["col_scale"], a["salient_idx"], a["residual_vals"],
                     a["residual_idx"])
    torch.cuda.synchronize()
    assert qt.qtea_device_status(layout) == 0
    return y, layout


def check(y, p, what, rows=None):
    y_ref, bound = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, rows=rows,
                               residual_fp8=p.residual_fp8)
    yy = y.cpu().numpy().astype(np.float64)
    if rows is not None:
        yy = yy[:, rows]
    err = np.abs(yy - y_ref)
    lim = REL * bound + ABS
    bad = np.argwhere(err > lim)
    assert bad.size == 0, f"{what}: {len(bad)} out of tolerance, worst normalised error {(err / lim).max():.3g}"
    return float((err / lim).max())


SHAPES = [  # N, K, s
    (4, 128, 0), (4, 128, 8), (12, 300, 16), (516, 1000, 32), (512, 1024, 32), (1000, 2048, 64),
    (1024, 4096, 120), (2052, 1536, 48), (520, 3000, 88), (4, 64, 4),
]


@pytest.mark.parametrize("N,K,s", SHAPES)
@pytest.mark.parametrize("fp8", [False, True])
def test_lut_parity_small(qt, N, K, s, fp8):
    p = synth.make_problem("lut", N, K, 1, s, seed=N + 3 * K + 7 * s + fp8, residual_fp8=fp8)
    y, _ = run(qt, p)
    check(y, p, f"N={N} K={K} s={s} fp8={fp8}")


@pytest.mark.parametrize("N,K,s", [(512, 1024, 1024), (256, 2048, 1000), (1024, 8192, 2048)])
def test_lut_dense_salient(qt, N, K, s):
    """Many salient entries per chunk (every column salient at K = 1024: one chunk takes all 1024)."""
    p = synth.make_problem("lut", N, K, 1, s, seed=5 * N + K + s)
    y, _ = run(qt, p)
    check(y, p, f"dense salient N={N} K={K} s={s}")


@pytest.mark.parametrize("matrix", range(7))
def test_lut_llama3_8b_layer(qt, matrix):
    p = synth.workload_problem("llama3_8b_layer", matrix)
    y, _ = run(qt, p)
    rng = np.random.default_rng(matrix)
    rows = np.unique(np.concatenate([[0, 1, 511, 512, p.N - 1], rng.integers(0, p.N, 64)])).astype(np.int32)
    worst = check(y, p, p.name, rows=rows)
    assert worst < 0.25


def test_lut_grouped_layer_and_bitwise_repeat(qt):
    ps = [synth.workload_problem("llama3_8b_layer", m) for m in range(7)]
    lays = [lut_layout(qt, p) for p in ps]
    probs = [dict(layout=l, **args(p)) for l, p in zip(lays, ps)]
    ys = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(lays[0]) == 0
    for m, (p, y) in enumerate(zip(ps, ys)):
        rows = np.arange(0, p.N, 97, dtype=np.int32)
        check(y, p, f"grouped {p.name}", rows=rows)
    ys2 = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    for y, y2 in zip(ys, ys2):
        assert torch.equal(y, y2)


@pytest.mark.parametrize("mags,sd", [([30000.0], 0.3), ([60000.0, 40000.0, 20000.0, 6000.0], 0.1)])
def test_lut_massive_activations(qt, mags, sd):
    """The table entries are fp32 sums of exact v*x products: no block-relative rounding."""
    p = synth.make_problem("lut", 1024, 4096, 1, 120, seed=700, x_std=sd)
    synth.plant_massive(p.x, 900, mags, 512, 1024)
    y, _ = run(qt, p)
    assert check(y, p, f"massive {mags}") < 0.25


def test_lut_matches_fixed_point_kernel_within_tolerance(qt):
    """The same base-3 layout through both decodes (the default table and QTEA_OPT_FIXED_POINT)."""
    p = synth.workload_problem("llama3_8b_layer", 1)
    y_lut, layout = run(qt, p)
    layout.set_options(qt.QTEA_OPT_FIXED_POINT)
    y_dp4a, _ = run(qt, p, layout)
    y_ref, bound = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx)
    lim = REL * bound + ABS
    assert np.all(np.abs(y_lut.cpu().numpy() - y_dp4a.cpu().numpy()) <= 2 * lim)
