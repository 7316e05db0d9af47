"""GPU parity: the CUDA library against the fp64 oracle on identical seeded inputs.

Pass rule (per output element): |y - y_ref| <= 1e-4 * sum_j |x_j * W^[o][j]| + 1e-6, the
bound computed by the oracle. Packing must be bit-identical to the oracle's packer.
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


class Dev:
    """Device copies of a synthetic problem plus its packed layout."""

    def __init__(self, qt, p: synth.Problem, act_bits: int = 24):
        self.p = p
        self.T = dev(p.T)
        self.layout = qt.qtea_pack_layout(self.T, n_salient=p.s)
        if act_bits != 24:
            self.layout.set_activation_precision(act_bits)
        self.x = dev(p.x.view(np.int16), torch.float16)
        self.alpha = dev(p.alpha.reshape(-1).view(np.int16), torch.float16)
        self.v = dev(p.v.view(np.int16), torch.float16)
        self.sal = dev(p.salient_idx) if p.s else None
        self.rv = dev(p.residual_vals.view(np.int16), torch.float16) if p.s else None
        self.ri = dev(p.residual_idx) if p.s else None

    def run(self, qt, x=None):
        y = qt.qtea_gemv(self.x if x is None else x, self.layout, self.alpha, self.v, self.sal, self.rv, self.ri)
        torch.cuda.synchronize()
        assert qt.qtea_device_status(self.layout) == 0
        return y.cpu().numpy().astype(np.float64)


def oracle_ref(p, rows=None, x=None):
    return oracle.gemv(p.x if x is None else x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals,
                       p.residual_idx, rows=rows)


def assert_within(y, y_ref, bound, what=""):
    err = np.abs(y - y_ref)
    lim = REL * bound + ABS
    bad = np.argwhere(err > lim)
    assert bad.size == 0, (f"{what}: {len(bad)} elements out of tolerance; worst normalised error "
                           f"{(err / lim).max():.3g} at {bad[0].tolist()}")
    return float((err / lim).max())


# ---------------------------------------------------------------- packing

@pytest.mark.parametrize("N,K", [(1, 1), (4, 64), (7, 100), (256, 512), (300, 1000), (1024, 4096)])
def test_pack_is_bit_identical_to_oracle(qt, N, K):
    T = synth.codes(N + K, 1, (N, K), 0.3, 0.4)
    lay = qt.qtea_pack_layout(dev(T))
    got = qt.packed_bytes(lay).cpu().numpy()
    assert np.array_equal(got, oracle.pack(T, "2bit"))
    assert lay.describe()["K_pad"] == -(-K // 64) * 64


@pytest.mark.parametrize("workload,matrix", [("tiny_1024", 0), ("llama3_8b_layer", 0), ("llama3_8b_layer", 1),
                                              ("llama3_8b_layer", 6), ("llama3_70b_layer", 4),
                                              ("llama3_70b_layer", 6)])
def test_batch1_kernel_serves_workload_shapes(qt, workload, matrix):
    """The workload shapes must run on the TMA stream-K kernel, not the general fallback."""
    p = synth.workload_problem(workload, matrix)
    lay = qt.qtea_pack_layout(dev(p.T), n_salient=p.s)
    assert lay.describe()["batch1_kernel"] == 1


def test_pack_rejects_invalid_codes(qt):
    T = synth.codes(1, 1, (64, 128), 0.3, 0.4)
    T[17, 33] = 2
    with pytest.raises(qt.QteaError) as e:
        qt.qtea_pack_layout(dev(T))
    assert e.value.status == qt.QTEA_ERR_BAD_CODES
    T[17, 33] = -128
    with pytest.raises(qt.QteaError):
        qt.qtea_pack_layout(dev(T))


# ---------------------------------------------------------------- small and ragged shapes, every M

SHAPES = [  # N, K, s: several tiles, ragged tails in both dimensions, s = 0 and s > 0
    (4, 64, 0), (4, 64, 8), (8, 100, 4), (256, 512, 16), (260, 520, 8), (1000, 1100, 32),
    (1024, 1024, 32), (2048, 4096, 120), (768, 3000, 88), (4096, 1536, 40),
]


@pytest.mark.parametrize("N,K,s", SHAPES)
@pytest.mark.parametrize("M", [1, 2, 5, 16])
def test_parity_small(qt, N, K, s, M):
    p = synth.make_problem("t", N, K, M, s, seed=N * 7 + K * 3 + s + M)
    d = Dev(qt, p)
    y = d.run(qt)
    y_ref, b = oracle_ref(p)
    assert_within(y, y_ref, b, f"N={N} K={K} s={s} M={M}")


DENSE_SALIENT = [  # more than 16 salient entries per unit (residual summed by the staging warps),
    # s not a multiple of 8 (scalar residual loads), every column salient
    (512, 1024, 400), (300, 2048, 100), (1024, 1024, 1024), (2048, 4096, 600), (4, 64, 64), (516, 700, 36),
]


@pytest.mark.parametrize("N,K,s", DENSE_SALIENT)
@pytest.mark.parametrize("M", [1, 3, 12])
def test_parity_dense_salient(qt, N, K, s, M):
    p = synth.make_problem("t", N, K, M, s, seed=N + 3 * K + 5 * s + M)
    d = Dev(qt, p)
    y = d.run(qt)
    y_ref, b = oracle_ref(p)
    assert_within(y, y_ref, b, f"N={N} K={K} s={s} M={M}")


@pytest.mark.parametrize("M", [2, 9])
def test_low_batch_unaligned_operands(qt, M):
    """x and v starting 2 bytes past a 16-byte boundary, K odd, residual values 2 bytes past an
    8-byte boundary (scalar residual loads)."""
    N, K, s = 516, 777, 12
    p = synth.make_problem("t", N, K, M, s, seed=40 + M)
    d = Dev(qt, p)

    def shifted(t):
        buf = torch.zeros(t.numel() + 1, dtype=t.dtype, device=t.device)
        buf[1:] = t.reshape(-1)
        return buf[1:].view(t.shape)

    x, v, rv = shifted(d.x), shifted(d.v), shifted(d.rv)
    assert x.data_ptr() % 16 == 2 and rv.data_ptr() % 8 == 2
    y = qt.qtea_gemv(x, d.layout, d.alpha, v, d.sal, rv, d.ri)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(d.layout) == 0
    y_ref, b = oracle_ref(p)
    assert_within(y.cpu().numpy().astype(np.float64), y_ref, b, f"unaligned M={M}")


def test_tiny_1024(qt):
    p = synth.workload_problem("tiny_1024", 0)
    d = Dev(qt, p)
    y = d.run(qt)
    y_ref, b = oracle_ref(p)
    worst = assert_within(y, y_ref, b, "tiny_1024")
    assert worst < 0.25  # keep a 4x margin on the tolerance


def test_zero_activation_gives_exact_zero(qt):
    p = synth.make_problem("t", 512, 2048, 1, 16, seed=1)
    p.x[:] = 0
    d = Dev(qt, p)
    assert np.all(d.run(qt) == 0.0)


def test_zero_residual_equals_ternary_only(qt):
    p = synth.make_problem("t", 1024, 2048, 1, 64, seed=2)
    p.residual_vals[:] = 0
    d = Dev(qt, p)
    y = d.run(qt)
    y0, b0 = oracle.gemv(p.x, p.T, p.alpha, p.v)
    assert_within(y, y0, b0, "zero residual")
    q = synth.make_problem("t", 1024, 2048, 1, 0, seed=2)
    dq = Dev(qt, q)
    assert np.array_equal(dq.run(qt), y)  # the zero residual contributes exactly nothing


def test_unit_vectors_extract_columns(qt):
    N, K = 512, 1024
    p = synth.make_problem("t", N, K, 1, 32, seed=3)
    d = Dev(qt, p)
    for k in [0, 511, 512, int(p.salient_idx[5]), K - 1]:
        x = np.zeros((1, K), np.uint16)
        x[0, k] = synth.f16_from_double(1.5)
        y = d.run(qt, dev(x.view(np.int16), torch.float16))
        y_ref, b = oracle_ref(p, x=x)
        assert_within(y, y_ref, b, f"e_{k}")


def test_outlier_activation_keeps_tolerance(qt):
    """A few huge activations in a block of small ones: per-block scaling keeps other blocks exact."""
    N, K = 1024, 4096
    p = synth.make_problem("t", N, K, 1, 120, seed=4)
    x = p.x.view(np.float16).astype(np.float32)
    x[0, [7, 1500, 3000]] = [3000.0, -2500.0, 1800.0]
    p.x = x.astype(np.float16).view(np.uint16).reshape(1, K)
    d = Dev(qt, p)
    y = d.run(qt)
    y_ref, b = oracle_ref(p)
    assert_within(y, y_ref, b, "outliers")


def test_bitwise_deterministic(qt):
    p = synth.make_problem("t", 4096, 4096, 1, 120, seed=5)
    d = Dev(qt, p)
    y1, y2 = d.run(qt), d.run(qt)
    assert np.array_equal(y1, y2)


def test_rejects_bad_arguments(qt):
    import ctypes
    p = synth.make_problem("t", 64, 128, 1, 8, seed=6)
    d = Dev(qt, p)
    lib = qt.load()
    y = torch.empty((1, 64), dtype=torch.float32, device="cuda")
    args = [d.x.data_ptr(), d.layout.handle, d.alpha.data_ptr(), d.v.data_ptr(), d.sal.data_ptr(), d.rv.data_ptr(),
            d.ri.data_ptr(), y.data_ptr()]
    assert lib.qtea_gemv(*args, 0, None) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_gemv(*args, 17, None) == qt.QTEA_ERR_INVALID_ARG
    bad = list(args)
    bad[7] = y.data_ptr() + 2  # misaligned y
    assert lib.qtea_gemv(*bad, 1, None) == qt.QTEA_ERR_INVALID_ARG
    bad = list(args)
    bad[4] = None  # missing salient indices with s > 0
    assert lib.qtea_gemv(*bad, 1, None) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_gemv(*args, 1, None) == qt.QTEA_OK
    torch.cuda.synchronize()


def test_empty_shapes(qt):
    lay = qt.qtea_pack_layout(torch.zeros((0, 64), dtype=torch.int8, device="cuda"))
    x = torch.zeros((1, 64), dtype=torch.float16, device="cuda")
    y = qt.qtea_gemv(x, lay, torch.zeros(0, dtype=torch.float16, device="cuda"),
                     torch.zeros(64, dtype=torch.float16, device="cuda"))
    assert y.shape == (1, 0)
    lay = qt.qtea_pack_layout(torch.zeros((8, 0), dtype=torch.int8, device="cuda"))
    y = qt.qtea_gemv(torch.zeros((2, 0), dtype=torch.float16, device="cuda"), lay,
                     torch.ones(8, dtype=torch.float16, device="cuda"), torch.zeros(0, dtype=torch.float16, device="cuda"))
    torch.cuda.synchronize()
    assert torch.all(y == 0)


# ---------------------------------------------------------------- full-size layer shapes (sampled rows)

def sample_rows(N, n=48, seed=0):
    rng = np.random.default_rng(seed)
    edge = [0, 1, 255, 256, 257, 511, 512, 513, N // 2, N - 513, N - 512, N - 257, N - 256, N - 2, N - 1]
    rows = sorted(set([r for r in edge if 0 <= r < N] + rng.integers(0, N, n).tolist()))
    return np.array(rows, np.int32)


@pytest.mark.parametrize("workload,matrix",
                         [("llama3_8b_layer", m) for m in range(7)] + [("llama3_70b_layer", m) for m in range(7)])
def test_full_size_layers_m1(qt, workload, matrix):
    p = synth.workload_problem(workload, matrix)
    d = Dev(qt, p)
    y = d.run(qt)
    rows = sample_rows(p.N, seed=matrix)
    y_ref, b = oracle_ref(p, rows=rows)
    assert_within(y[:, rows], y_ref, b, p.name)


@pytest.mark.parametrize("matrix", range(7))
@pytest.mark.parametrize("M", [1, 2, 4, 8, 16])
def test_full_size_qwen3_14b_batch_sweep(qt, matrix, M):
    p = synth.workload_problem("qwen3_14b_layer", matrix, M=M)
    d = Dev(qt, p)
    y = d.run(qt)
    rows = sample_rows(p.N, n=16, seed=matrix + M)
    y_ref, b = oracle_ref(p, rows=rows)
    assert_within(y[:, rows], y_ref, b, f"{p.name} M={M}")


# ---------------------------------------------------------------- grouped launches

def problem_dict(d):
    return dict(x=d.x, layout=d.layout, row_scale=d.alpha, col_scale=d.v, salient_idx=d.sal, residual_vals=d.rv,
                residual_idx=d.ri)


@pytest.mark.parametrize("n", [1, 3, 8, 11])
def test_grouped_matches_oracle(qt, n):
    shapes = [(4, 64, 0), (1024, 4096, 120), (260, 520, 8), (2048, 1536, 48), (1000, 1100, 32), (516, 8192, 248),
              (64, 128, 8), (4096, 1024, 32), (8, 100, 4), (1536, 2048, 64), (512, 512, 16)]
    ps = [synth.make_problem("g", N, K, 1, s, seed=100 * i + n) for i, (N, K, s) in enumerate(shapes[:n])]
    ds = [Dev(qt, p) for p in ps]
    ys = qt.qtea_gemv_grouped([problem_dict(d) for d in ds])
    torch.cuda.synchronize()
    assert qt.qtea_device_status(ds[0].layout) == 0
    for p, y in zip(ps, ys):
        y_ref, b = oracle_ref(p)
        assert_within(y.cpu().numpy().astype(np.float64), y_ref, b, f"grouped {p.N}x{p.K}")


def test_grouped_llama3_8b_layer(qt):
    ps = [synth.workload_problem("llama3_8b_layer", m) for m in range(7)]
    ds = [Dev(qt, p) for p in ps]
    ys = qt.qtea_gemv_grouped([problem_dict(d) for d in ds])
    torch.cuda.synchronize()
    for m, (p, y) in enumerate(zip(ps, ys)):
        rows = sample_rows(p.N, n=24, seed=m)
        y_ref, b = oracle_ref(p, rows=rows)
        assert_within(y.cpu().numpy().astype(np.float64)[:, rows], y_ref, b, p.name)
    # a repeated grouped call reproduces its result bit for bit (the split of tiles over CTAs,
    # hence the summation order, depends on the group, so single calls may differ in rounding)
    ys2 = qt.qtea_gemv_grouped([problem_dict(d) for d in ds])
    torch.cuda.synchronize()
    for y, y2 in zip(ys, ys2):
        assert torch.equal(y, y2)


@pytest.mark.parametrize("layer", [0, 17, 31])
def test_grouped_llama3_8b_stack_layers(qt, layer):
    """Layers of the 32-layer stack (independent seeds per layer), as the benchmark launches them."""
    ps = [synth.workload_problem("llama3_8b_32layer_stack", m, layer=layer) for m in range(7)]
    ds = [Dev(qt, p) for p in ps]
    ys = qt.qtea_gemv_grouped([problem_dict(d) for d in ds])
    torch.cuda.synchronize()
    assert qt.qtea_device_status(ds[0].layout) == 0
    for m, (p, y) in enumerate(zip(ps, ys)):
        rows = sample_rows(p.N, n=12, seed=layer * 7 + m)
        y_ref, b = oracle_ref(p, rows=rows)
        assert_within(y.cpu().numpy().astype(np.float64)[:, rows], y_ref, b, f"{p.name} layer {layer}")


def test_grouped_rejects_shared_layout_and_mixed_batch(qt):
    p = synth.make_problem("g", 64, 128, 1, 8, seed=1)
    d = Dev(qt, p)
    with pytest.raises(qt.QteaError):
        qt.qtea_gemv_grouped([problem_dict(d), problem_dict(d)])
    q = synth.make_problem("g", 64, 128, 2, 8, seed=2)
    e = Dev(qt, q)
    with pytest.raises(ValueError):
        qt.qtea_gemv_grouped([problem_dict(d), problem_dict(e)])


def test_grouped_batch2_uses_general_path(qt):
    ps = [synth.make_problem("g", N, K, 2, s, seed=i) for i, (N, K, s) in enumerate([(256, 512, 8), (100, 200, 0)])]
    ds = [Dev(qt, p) for p in ps]
    ys = qt.qtea_gemv_grouped([problem_dict(d) for d in ds])
    torch.cuda.synchronize()
    for p, y in zip(ps, ys):
        y_ref, b = oracle_ref(p)
        assert_within(y.cpu().numpy().astype(np.float64), y_ref, b, "grouped M=2")


# ---------------------------------------------------------------- 16-bit activation mode

@pytest.mark.parametrize("workload,matrix", [("tiny_1024", 0), ("llama3_8b_layer", 1), ("llama3_8b_layer", 4),
                                              ("llama3_8b_layer", 6), ("qwen3_14b_layer", 0), ("qwen3_14b_layer", 6),
                                              ("llama3_70b_layer", 1), ("llama3_70b_layer", 6)])
def test_fast_mode_keeps_a_4x_margin(qt, workload, matrix):
    p = synth.workload_problem(workload, matrix)
    d = Dev(qt, p, act_bits=16)
    y = d.run(qt)
    rows = sample_rows(p.N, n=64, seed=synth.WORKLOADS[workload]["seed_base"] // 100 + matrix)
    y_ref, b = oracle_ref(p, rows=rows)
    worst = assert_within(y[:, rows], y_ref, b, f"16-bit {p.name}")
    assert worst < 0.25


def test_fast_mode_outliers_fall_back_to_24_bits(qt):
    N, K = 1024, 4096
    p = synth.make_problem("t", N, K, 1, 120, seed=4)
    x = p.x.view(np.float16).astype(np.float32)
    x[0, [7, 1500, 3000]] = [3000.0, -2500.0, 1800.0]
    p.x = x.astype(np.float16).view(np.uint16).reshape(1, K)
    d = Dev(qt, p, act_bits=16)
    y = d.run(qt)
    y_ref, b = oracle_ref(p)
    assert_within(y, y_ref, b, "16-bit with outliers")


def test_activation_precision_argument(qt):
    p = synth.make_problem("t", 64, 128, 1, 8, seed=6)
    d = Dev(qt, p)
    with pytest.raises(qt.QteaError):
        d.layout.set_activation_precision(8)
    d.layout.set_activation_precision(16)  # K < 1024: stays 24-bit, still within tolerance
    y = d.run(qt)
    y_ref, b = oracle_ref(p)
    assert_within(y, y_ref, b, "small K in 16-bit mode")
