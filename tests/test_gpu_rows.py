"""GPU parity of the row-resident batch-1 kernel (whole rows per CTA, codes fetched before the grid
dependency wait) against the fp64 oracle.

The kernel takes a batch-1 call when all of its 2-bit, one-alpha-per-row problems fit one launch of
it (at most 32 rows per CTA, one or two CTAs per SM; a wide launch, K above 4096 or more than 256
salient columns, one CTA per SM, K up to 8192, up to 512 salient columns); larger calls take the
stream-K kernel. Pass rule (per output element): |y - y_ref| <= 1e-4 * sum_j |x_j * W^[o][j]| + 1e-6,
the oracle's bound. Shapes cover one, two and four lanes per row, a CTA whose last 8-row block is
half empty, ragged K (a chunk shorter than 512 columns), one-CTA problems, every column salient,
warps with one to four chunks, grouped calls that split the SMs between problems, unaligned
activations (scalar staging loads) and massive activations.
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


def f16(a):
    return dev(np.ascontiguousarray(a).view(np.int16), torch.float16)


def args(p, x_offset=0):
    """Device arguments of problem p; with x_offset > 0, x and v start x_offset elements into a
    larger buffer (2-byte aligned only: the staging takes its scalar loads)."""
    if x_offset:
        xb = torch.zeros(p.K + x_offset, dtype=torch.float16, device="cuda")
        vb = torch.zeros(p.K + x_offset, dtype=torch.float16, device="cuda")
        xb[x_offset:] = f16(p.x.reshape(-1))
        vb[x_offset:] = f16(p.v)
        x, v = xb[x_offset:].view(1, p.K), vb[x_offset:]
    else:
        x, v = f16(p.x), f16(p.v)
    return dict(x=x, row_scale=f16(p.alpha.reshape(-1)), col_scale=v,
                salient_idx=dev(p.salient_idx) if p.s else None,
                residual_vals=f16(p.residual_vals) if p.s else None,
                residual_idx=dev(p.residual_idx) if p.s else None)


def layout_of(qt, p, stream_k=False, bits=16):
    lay = qt.qtea_pack_layout(dev(p.T), n_salient=p.s)
    if stream_k:
        lay.set_options(qt.QTEA_OPT_STREAM_K)
    if bits != 16:
        lay.set_activation_precision(bits)
    return lay


def run(qt, p, lay, x_offset=0):
    a = args(p, x_offset)
    y = qt.qtea_gemv(a["x"], lay, a["row_scale"], a["col_scale"], a["salient_idx"], a["residual_vals"],
                     a["residual_idx"])
    torch.cuda.synchronize()
    assert qt.qtea_device_status(lay) == 0
    return y


def check(y, p, what, rows=None):
    y_ref, bound = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, rows=rows)
    yy = y.cpu().numpy().astype(np.float64)
    if rows is not None:
        yy = yy[:, rows]
    err = np.abs(yy - y_ref)
    lim = REL * bound + ABS
    bad = np.argwhere(err > lim)
    assert bad.size == 0, f"{what}: {len(bad)} out of tolerance, worst normalised error {(err / lim).max():.3g}"
    return float((err / lim).max())


def test_eligibility(qt):
    p = synth.make_problem("rows", 64, 256, 1, 8, seed=1)
    lay = layout_of(qt, p)
    assert lay.describe()["rows_kernel"] == 1
    lay.set_options(qt.QTEA_OPT_STREAM_K)
    assert lay.describe()["rows_kernel"] == 0 and lay.describe()["batch1_kernel"] == 1
    g = synth.make_problem("rows", 64, 256, 1, 8, seed=1, group_size=128)
    assert qt.qtea_pack_layout(dev(g.T), n_salient=8, group_size=128).describe()["rows_kernel"] == 0
    assert qt.qtea_pack_layout(dev(p.T), n_salient=8, fmt=qt.QTEA_FMT_BASE3).describe()["rows_kernel"] == 0


def test_plan_small_calls_rows_large_calls_stream_k(qt):
    """Which batch-1 form a call takes: q, k, v, o of the Llama3-8B layer alone and q, k, v together
    fit the row-resident launch; gate_proj (14336 rows, more than 32 per CTA), down_proj (K = 14336,
    beyond the wide launch's 8192) and the whole layer in one call take the stream-K launch, as does
    a layout pinned to it."""
    ps = [synth.workload_problem("llama3_8b_layer", m) for m in range(7)]
    lays = [layout_of(qt, p) for p in ps]
    probs = [dict(layout=l, **args(p)) for l, p in zip(lays, ps)]
    for m in (0, 1, 2, 3):
        assert qt.qtea_gemv_plan([probs[m]]) == ["rows"]
    assert qt.qtea_gemv_plan(probs[:3]) == ["rows"] * 3
    assert qt.qtea_gemv_plan([probs[4]]) == ["stream_k"]
    assert qt.qtea_gemv_plan([probs[6]]) == ["stream_k"]
    assert qt.qtea_gemv_plan(probs) == ["stream_k"] * 7
    lays[1].set_options(qt.QTEA_OPT_STREAM_K)
    assert qt.qtea_gemv_plan(probs[:3]) == ["stream_k"] * 3


SHAPES = [  # N, K, s
    (4, 128, 0), (4, 128, 8), (8, 64, 0), (12, 300, 16), (4, 64, 4), (3, 100, 0), (1, 1, 0), (7, 7, 0),
    (516, 1000, 32), (512, 1024, 32), (1000, 2048, 64), (1024, 4096, 120), (2052, 1536, 48), (520, 3000, 88),
    (64, 3584, 104), (9728, 4096, 120), (4864, 2048, 64), (4096, 4096, 120), (19456, 4096, 128),
]


@pytest.mark.parametrize("N,K,s", SHAPES)
def test_rows_parity_shapes(qt, N, K, s):
    p = synth.make_problem("rows", N, K, 1, s, seed=N + 5 * K + 11 * s)
    y = run(qt, p, layout_of(qt, p))
    check(y, p, f"N={N} K={K} s={s}")


@pytest.mark.parametrize("N,K,s", [(512, 256, 256), (64, 256, 256), (256, 2048, 256), (1024, 4096, 248)])
def test_rows_dense_salient(qt, N, K, s):
    p = synth.make_problem("rows", N, K, 1, s, seed=3 * N + K + s)
    check(run(qt, p, layout_of(qt, p)), p, f"dense salient N={N} K={K} s={s}")


WIDE_SHAPES = [  # N, K, s: more than one chunk per warp, or more than 256 salient columns
    (512, 4608, 32), (1004, 8000, 64), (2052, 5000, 100), (4, 8192, 8), (256, 8192, 512),
    (4864, 8192, 432), (1024, 4096, 300), (256, 512, 512), (8, 7000, 264),
]


@pytest.mark.parametrize("N,K,s", WIDE_SHAPES)
def test_rows_wide_parity_shapes(qt, N, K, s):
    """Wide launches: warps with two chunks (the next chunk's x and v loaded during a decode), a
    ragged last chunk, one to four lanes per row, up to 512 salient columns in registers."""
    p = synth.make_problem("rows/wide", N, K, 1, s, seed=7 * N + K + 13 * s)
    lay = layout_of(qt, p)
    assert lay.describe()["rows_kernel"] == 1
    assert qt.qtea_gemv_plan([dict(layout=lay, **args(p))]) == ["rows"]
    y = run(qt, p, lay)
    rows = None if N * K <= 1 << 24 else np.unique(np.concatenate(
        [np.arange(0, N, 37), [0, 1, 7, 8, 31, 32, N - 1]])).astype(np.int32)
    check(y, p, f"wide N={N} K={K} s={s}", rows=rows)


def test_rows_wide_limits(qt):
    """Past the wide launch's limits the stream-K kernel serves the call: more than 32 rows per CTA
    with one CTA per SM, more than 16 chunks, more than 512 salient columns."""
    sm = torch.cuda.get_device_properties(0).multi_processor_count
    for N, K, s in ((8 * (4 * sm + 1), 4608, 8), (64, 8704, 8), (64, 4096, 520)):
        p = synth.make_problem("rows/limits", N, K, 1, s, seed=N + K + s)
        lay = layout_of(qt, p)
        assert qt.qtea_gemv_plan([dict(layout=lay, **args(p))]) == ["stream_k"], (N, K, s)
        rows = np.unique(np.concatenate([np.arange(0, N, 97), [N - 1]])).astype(np.int32)
        check(run(qt, p, lay), p, f"stream-K beyond the wide limits N={N} K={K} s={s}", rows=rows)


@pytest.mark.parametrize("workload,matrix", [("qwen3_14b_layer", 1), ("llama3_70b_layer", 2)])
def test_rows_wide_workload_calls(qt, workload, matrix):
    """k_proj of Qwen3-14B (K = 5120) and v_proj of Llama3-70B (K = 8192) alone: wide launches,
    sampled rows."""
    p = synth.workload_problem(workload, matrix)
    lay = layout_of(qt, p)
    assert qt.qtea_gemv_plan([dict(layout=lay, **args(p))]) == ["rows"]
    y = run(qt, p, lay)
    rows = np.unique(np.concatenate([np.arange(0, p.N, 29), [0, 7, 8, p.N - 1]])).astype(np.int32)
    assert check(y, p, f"{workload} {p.name}", rows=rows) < 0.25


def test_rows_wide_grouped_call(qt):
    """Two wide problems and a narrow one in one launch (one CTA per SM): results match the oracle
    and repeat bitwise."""
    ps = [synth.make_problem("rows/wg", N, K, 1, s, seed=N + K + s)
          for N, K, s in ((512, 8192, 64), (256, 4096, 300), (128, 2048, 16))]
    lays = [layout_of(qt, p) for p in ps]
    probs = [dict(layout=l, **args(p)) for l, p in zip(lays, ps)]
    assert qt.qtea_gemv_plan(probs) == ["rows"] * 3
    ys = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(lays[0]) == 0
    for p, y in zip(ps, ys):
        check(y, p, f"wide grouped {p.name} N={p.N} K={p.K}")
    ys2 = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    for y, y2 in zip(ys, ys2):
        assert torch.equal(y, y2)


@pytest.mark.parametrize("N,K,s", [(516, 1000, 32), (4096, 4096, 120), (516, 7000, 40)])
def test_rows_unaligned_activations(qt, N, K, s):
    p = synth.make_problem("rows", N, K, 1, s, seed=N + K)
    check(run(qt, p, layout_of(qt, p), x_offset=1), p, f"x at an odd offset N={N} K={K}")


@pytest.mark.parametrize("matrix", [0, 1, 2, 3])
def test_rows_llama3_8b_layer(qt, matrix):
    """q, k, v and o of the Llama3-8B layer, each alone (one call), sampled rows."""
    p = synth.workload_problem("llama3_8b_layer", matrix)
    lay = layout_of(qt, p)
    y = run(qt, p, lay)
    rng = np.random.default_rng(matrix)
    rows = np.unique(np.concatenate([[0, 1, 7, 8, 31, 32, 63, p.N - 1], rng.integers(0, p.N, 96)])).astype(np.int32)
    assert check(y, p, p.name, rows=rows) < 0.25


@pytest.mark.parametrize("workload,mats", [("llama3_8b_layer", (0, 1, 2)), ("llama3_8b_layer", (3,)),
                                           ("llama3_8b_layer", (1, 2, 3))])
def test_rows_grouped_calls(qt, workload, mats):
    """Grouped calls the decode stack makes (q, k, v together; o alone): the SMs are split between
    the problems; results match the oracle and repeat bitwise."""
    ps = [synth.workload_problem(workload, m) for m in mats]
    lays = [layout_of(qt, p) for p in ps]
    probs = [dict(layout=l, **args(p)) for l, p in zip(lays, ps)]
    ys = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(lays[0]) == 0
    for p, y in zip(ps, ys):
        rows = np.unique(np.concatenate([np.arange(0, p.N, 53), [p.N - 1]])).astype(np.int32)
        check(y, p, f"grouped {p.name}", rows=rows)
    ys2 = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    for y, y2 in zip(ys, ys2):
        assert torch.equal(y, y2)


@pytest.mark.parametrize("bits", [16, 24])
def test_rows_matches_stream_k_kernel(qt, bits):
    """The same layout through both batch-1 forms: both within tolerance of the oracle, and of each
    other within twice the tolerance."""
    p = synth.workload_problem("llama3_8b_layer", 0)
    lay = layout_of(qt, p, bits=bits)
    y_rows = run(qt, p, lay)
    lay.set_options(qt.QTEA_OPT_STREAM_K)
    y_sk = run(qt, p, lay)
    y_ref, bound = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx)
    lim = REL * bound + ABS
    for y in (y_rows, y_sk):
        assert np.all(np.abs(y.cpu().numpy() - y_ref) <= lim)
    assert np.all(np.abs(y_rows.cpu().numpy() - y_sk.cpu().numpy()) <= 2 * lim)


@pytest.mark.parametrize("mags,sd", [([30000.0], 0.3), ([60000.0, 40000.0, 20000.0, 6000.0], 0.1),
                                     ([3000.0, 60000.0], 0.2)])
@pytest.mark.parametrize("bits", [16, 24])
def test_rows_massive_activations(qt, mags, sd, bits):
    """Values of 3e3 to 6e4 among N(0, 0.1 to 0.3) activations in one 512-column chunk: taken out of
    the fixed-point planes and added exactly; rows whose code is 0 at those columns are checked."""
    p = synth.make_problem("rows/massive", 1024, 4096, 1, 120, seed=700, x_std=sd)
    cols = synth.plant_massive(p.x, 900, mags, 512, 1024)
    y = run(qt, p, layout_of(qt, p, bits=bits))
    assert np.any(p.T[:, cols[0]] == 0)
    assert check(y, p, f"massive {mags} {bits}-bit") < 0.25
