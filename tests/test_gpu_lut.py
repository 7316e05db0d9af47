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


def paper_args(p, bias):
    f16 = lambda a: dev(np.ascontiguousarray(a).view(np.int16), torch.float16)
    if bias:
        sc = np.stack([p.alpha.reshape(p.N, -1), p.beta.reshape(p.N, -1)], axis=-1).reshape(-1)
    else:
        sc = p.alpha.reshape(-1)
    a = args(p)
    a["row_scale"] = f16(sc)
    return a


def run_grouped(qt, p, bias, fixed=False):
    layout = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, group_size=p.group_size or p.K, fmt=qt.QTEA_FMT_BASE3)
    opts = (qt.QTEA_OPT_BIAS if bias else 0) | (qt.QTEA_OPT_RESIDUAL_FP8 if p.residual_fp8 else 0)
    layout.set_options(opts | (qt.QTEA_OPT_FIXED_POINT if fixed else 0))
    a = paper_args(p, bias)
    y = qt.qtea_gemv(a["x"], layout, a["row_scale"], a["col_scale"], a["salient_idx"], a["residual_vals"],
                     a["residual_idx"])
    torch.cuda.synchronize()
    assert qt.qtea_device_status(layout) == 0
    return y


def check_grouped(y, p, bias, what, rows=None):
    y_ref, bound = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx,
                               beta=p.beta if bias else None, group_size=p.group_size or p.K, rows=rows,
                               residual_fp8=p.residual_fp8)
    yy = y.cpu().numpy().astype(np.float64)
    if rows is not None:
        yy = yy[:, rows]
    err = np.abs(yy - y_ref)
    lim = REL * bound + ABS
    assert np.all(err <= lim), f"{what}: worst normalised error {(err / lim).max():.3g}"
    return float((err / lim).max())


@pytest.mark.parametrize("N,K,s", [(4, 128, 4), (12, 300, 16), (516, 1000, 32), (1024, 1100, 40), (2048, 4096, 120)])
@pytest.mark.parametrize("group,bias,fp8", [(128, True, True), (128, False, False), (128, True, False), (0, True, True)])
def test_lut_scale_groups(qt, N, K, s, group, bias, fp8):
    """The paper's storage through the table: alpha (and beta) per 128-column group, or one (alpha,
    beta) pair per row (group 0 = K); K = 1100 leaves a last chunk of one block."""
    p = synth.make_problem("lutg", N, K, 1, s, seed=N + K + s + group + 2 * bias + fp8, group_size=group,
                           beta_std=0.002 if bias else 0.0, residual_fp8=fp8)
    y = run_grouped(qt, p, bias)
    check_grouped(y, p, bias, f"N={N} K={K} s={s} group={group} bias={bias} fp8={fp8}")


@pytest.mark.parametrize("matrix", range(7))
def test_lut_paper_storage_llama3_8b_layer(qt, matrix):
    """The Llama3-8B layer in the paper's storage (base-3, alpha and beta per 128 columns, FP8
    residual): the table decode, and within tolerance of the fixed-point kernel on the same layout."""
    p = synth.paper_problem("llama3_8b_layer", matrix)
    y = run_grouped(qt, p, True)
    rows = np.sort(np.random.default_rng(matrix).choice(p.N, size=48, replace=False)).astype(np.int32)
    assert check_grouped(y, p, True, p.name, rows=rows) < 0.25
    y_fixed = run_grouped(qt, p, True, fixed=True)
    check_grouped(y_fixed, p, True, p.name + " fixed point", rows=rows)


def test_lut_grouped_call_mixes_variants(qt):
    """One grouped call with base-3 problems with and without scale groups (two launches) and a
    2-bit problem: each result matches the oracle."""
    ps = [synth.paper_problem("llama3_8b_layer", 1), synth.workload_problem("llama3_8b_layer", 2),
          synth.make_problem("g", 1024, 2048, 1, 64, seed=3, group_size=128, beta_std=0.002)]
    bias = [True, False, True]
    fmts = [qt.QTEA_FMT_BASE3, qt.QTEA_FMT_BASE3, qt.QTEA_FMT_BASE3]
    probs, lays = [], []
    for p, b, f in zip(ps, bias, fmts):
        lay = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, group_size=p.group_size or p.K, fmt=f)
        lay.set_options((qt.QTEA_OPT_BIAS if b else 0) | (qt.QTEA_OPT_RESIDUAL_FP8 if p.residual_fp8 else 0))
        lays.append(lay)
        probs.append(dict(layout=lay, **paper_args(p, b)))
    q2 = synth.workload_problem("llama3_8b_layer", 0)
    lay2 = qt.qtea_pack_layout(dev(q2.T), n_salient=q2.s)
    probs.append(dict(layout=lay2, **args(q2)))
    ys = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    for p, b, y in zip(ps, bias, ys):
        rows = np.arange(0, p.N, 37, dtype=np.int32)
        check_grouped(y, p, b, "mixed " + p.name, rows=rows)
    check(ys[3], q2, "mixed 2-bit", rows=np.arange(0, q2.N, 37, dtype=np.int32))
