"""GPU parity for layouts in the paper's own storage (Sec. 3.3 Eq. 4, Sec. 3.5, Sec. 4.1):
base-3 codes, alpha and beta per row and group of 128 columns, FP8 E4M3 residual values.

Same pass rule as test_gpu_parity: |y - y_ref| <= 1e-4 * sum_j |x_j * W^[o][j]| + 1e-6 per output
element, W^ including beta and the residual; base-3 packing bit-identical to the oracle's packer.
"""
import itertools

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


def scales(p, bias):
    """row_scale as the ABI wants it: [N][G] alpha, or [N][G][2] (alpha, beta) pairs."""
    if not bias:
        return p.alpha.reshape(-1)
    return np.stack([p.alpha.reshape(p.N, -1), p.beta.reshape(p.N, -1)], axis=-1).reshape(-1)


def run_paper(qt, p, fmt, bias, M=None):
    layout = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, group_size=p.group_size or p.K, fmt=fmt)
    opts = (qt.QTEA_OPT_BIAS if bias else 0) | (qt.QTEA_OPT_RESIDUAL_FP8 if p.residual_fp8 else 0)
    layout.set_options(opts)
    batch1 = fmt == qt.QTEA_FMT_2BIT and not p.residual_fp8  # 2-bit codes with fp16 residual values
    assert layout.describe()["batch1_kernel"] == int(batch1) and layout.describe()["options"] == opts
    x = p.x if M is None else p.x[:M]
    rv = dev(p.residual_vals) if p.residual_fp8 else dev(p.residual_vals.view(np.int16), torch.float16)
    y = qt.qtea_gemv(dev(x.view(np.int16), torch.float16), layout, dev(scales(p, bias).view(np.int16), torch.float16),
                     dev(p.v.view(np.int16), torch.float16), dev(p.salient_idx) if p.s else None,
                     rv if p.s else None, dev(p.residual_idx) if p.s else None)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(layout) == 0
    return y.cpu().numpy().astype(np.float64), layout


def reference(p, bias, rows=None, M=None):
    x = p.x if M is None else p.x[:M]
    return oracle.gemv(x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx,
                       beta=p.beta if bias else None, group_size=p.group_size or p.K, rows=rows,
                       residual_fp8=p.residual_fp8)


def assert_within(y, y_ref, bound, what=""):
    err = np.abs(y - y_ref)
    lim = REL * bound + ABS
    bad = np.argwhere(err > lim)
    assert bad.size == 0, (f"{what}: {len(bad)} elements out of tolerance; worst normalised error "
                           f"{(err / lim).max():.3g} at {bad[0].tolist()}")
    return float((err / lim).max())


@pytest.mark.parametrize("N,K", [(4, 128), (8, 1), (12, 300), (64, 1024), (33, 5)])
def test_base3_pack_is_bit_identical_to_oracle(qt, N, K):
    T = synth.codes(N * 1000 + K, 1, (N, K), 0.3, 0.4)
    layout = qt.qtea_pack_layout(dev(T), fmt=qt.QTEA_FMT_BASE3)
    d = layout.describe()
    assert d["K_pad"] == -(-K // 128) * 128 and d["packed_bytes"] == N * (-(-K // 128)) * 26
    got = qt.packed_bytes(layout)
    torch.cuda.synchronize()
    assert np.array_equal(got.cpu().numpy(), oracle.pack(T, "base3").reshape(-1))


def test_base3_pack_rejects_invalid_codes(qt):
    T = np.zeros((4, 256), np.int8)
    T[2, 200] = 2
    with pytest.raises(qt.QteaError) as e:
        qt.qtea_pack_layout(dev(T), fmt=qt.QTEA_FMT_BASE3)
    assert e.value.status == qt.QTEA_ERR_BAD_CODES


@pytest.mark.parametrize("fmt,group,bias,fp8", list(itertools.product([0, 1], [0, 128], [0, 1], [0, 1])))
def test_paper_storage_parity_small(qt, fmt, group, bias, fp8):
    """Every combination of code format, scale groups, beta and FP8 residual, K ragged against both
    the 128-column groups and the 64-column 2-bit padding, batch sizes 1, 3 and 16."""
    N, K, s = 64, 300, 16
    p = synth.make_problem("t", N, K, 16, s, seed=1 + fmt + 2 * bool(group) + 4 * bias + 8 * fp8,
                           group_size=group, beta_std=0.002 if bias else 0.0, residual_fp8=bool(fp8))
    for M in (1, 3, 16):
        y, _ = run_paper(qt, p, fmt, bias, M=M)
        y_ref, b = reference(p, bias, M=M)
        assert_within(y, y_ref, b, f"fmt {fmt} group {group} bias {bias} fp8 {fp8} M {M}")


def test_options_switch_a_default_layout_to_the_paper_path(qt):
    """A 2-bit, one-alpha-per-row layout with QTEA_OPT_BIAS reads (alpha, beta) pairs (on the batch-1
    kernel's grouped variant); FP8 residual values move it to the low-batch kernel; clearing the
    options returns it to the plain batch-1 kernel."""
    N, K = 256, 1024
    p = synth.make_problem("t", N, K, 1, 32, seed=5, beta_std=0.002)
    y, layout = run_paper(qt, p, qt.QTEA_FMT_2BIT, True)
    y_ref, b = reference(p, True)
    assert_within(y, y_ref, b, "2-bit with beta")
    assert layout.describe()["batch1_kernel"] == 1
    layout.set_options(qt.QTEA_OPT_RESIDUAL_FP8)
    assert layout.describe()["batch1_kernel"] == 0
    layout.set_options(0)
    assert layout.describe()["batch1_kernel"] == 1
    layout.set_options(qt.QTEA_OPT_FIXED_POINT)  # a base-3 choice: a 2-bit layout stays on the batch-1 kernel
    assert layout.describe()["batch1_kernel"] == 1
    with pytest.raises(qt.QteaError):
        layout.set_options(16)


@pytest.mark.parametrize("matrix", range(7))
@pytest.mark.parametrize("M", [1, 4])
def test_paper_storage_llama3_8b_layer(qt, matrix, M):
    """The Llama3-8B layer GEMVs in the paper's storage (base-3, 128-column groups with beta, FP8
    residual), on 48 sampled output rows."""
    p = synth.paper_problem("llama3_8b_layer", matrix, M=M)
    y, _ = run_paper(qt, p, qt.QTEA_FMT_BASE3, True)
    rows = np.sort(np.random.default_rng(matrix).choice(p.N, size=48, replace=False)).astype(np.int32)
    y_ref, b = reference(p, True, rows=rows)
    assert_within(y[:, rows], y_ref, b, p.name)


@pytest.mark.parametrize("fp8", [0, 1])
@pytest.mark.parametrize("bias", [0, 1])
@pytest.mark.parametrize("N,K,s", [(512, 2048, 24), (516, 3072, 40), (1024, 1024, 0), (260, 1536, 7)])
def test_group_scales_through_the_tensor_core_kernel(qt, N, K, s, bias, fp8):
    """2-bit codes with alpha (and beta) per 128-column group, fp16 or FP8 residual values, row_scale
    rows a multiple of 16 bytes (the shapes the tensor-core kernel takes): batch 1, 5 and 16, several
    tiles, ragged N, s not a multiple of 4 (byte-wise residual loads and tails)."""
    p = synth.make_problem("t", N, K, 16, s, seed=N + K + s + 7 * bias + 13 * fp8, group_size=128,
                           beta_std=0.002 if bias else 0.0, residual_fp8=bool(fp8))
    for M in (1, 5, 16):
        y, _ = run_paper(qt, p, qt.QTEA_FMT_2BIT, bias, M=M)
        y_ref, b = reference(p, bias, M=M)
        assert_within(y, y_ref, b, f"N {N} K {K} s {s} bias {bias} fp8 {fp8} M {M}")


@pytest.mark.parametrize("M", [1, 4, 16])
def test_fp8_residual_one_alpha_per_row_tensor_core_kernel(qt, M):
    """FP8 E4M3 residual with one alpha per row (the tensor-core kernel's helpers convert every E4M3
    value exactly), dense salient set, ragged N."""
    p = synth.make_problem("t", 1028, 2048, 16, 200, seed=77 + M, residual_fp8=True)
    y, _ = run_paper(qt, p, qt.QTEA_FMT_2BIT, False, M=M)
    y_ref, b = reference(p, False, M=M)
    assert_within(y, y_ref, b, f"fp8 M {M}")


def test_group_scales_llama3_8b_layer_2bit(qt):
    """The Llama3-8B layer with 2-bit codes, alpha and beta per 128-column group and fp16 residual, at
    batch 4, grouped in one call, on sampled rows."""
    ps = [synth.make_problem("g", N, K, 4, s, seed=3000 + m, group_size=128, beta_std=0.002)
          for m, (N, K, s) in enumerate([(4096, 4096, 120), (1024, 4096, 120), (14336, 4096, 120),
                                         (4096, 14336, 432)])]
    probs, lays = [], []
    for p in ps:
        lay = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, group_size=128, fmt=qt.QTEA_FMT_2BIT)
        lay.set_options(qt.QTEA_OPT_BIAS)
        lays.append(lay)
        probs.append(dict(x=dev(p.x.view(np.int16), torch.float16), layout=lay,
                          row_scale=dev(scales(p, True).view(np.int16), torch.float16),
                          col_scale=dev(p.v.view(np.int16), torch.float16), salient_idx=dev(p.salient_idx),
                          residual_vals=dev(p.residual_vals.view(np.int16), torch.float16),
                          residual_idx=dev(p.residual_idx)))
    ys = qt.qtea_gemv_grouped(probs)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(lays[0]) == 0
    for m, (p, y) in enumerate(zip(ps, ys)):
        rows = np.sort(np.random.default_rng(m).choice(p.N, size=32, replace=False)).astype(np.int32)
        y_ref, b = reference(p, True, rows=rows)
        assert_within(y.cpu().numpy().astype(np.float64)[:, rows], y_ref, b, f"{p.N}x{p.K}")


@pytest.mark.parametrize("M", [1, 3, 16])
def test_grouped_call_mixing_storage_formats(qt, M):
    """One grouped call over the library's own layouts, 2-bit layouts with scale groups (one kernel
    variant per launch, so the call splits), an FP8 residual and a base-3 layout (the general
    kernel): every y against the oracle."""
    specs = [  # (N, K, s, fmt, group, bias, fp8)
        (512, 2048, 24, 0, 0, 0, 0), (516, 2048, 16, 0, 128, 1, 0), (256, 1024, 8, 0, 0, 0, 0),
        (260, 3072, 12, 0, 128, 0, 1), (128, 1024, 8, 1, 128, 1, 1), (64, 300, 4, 0, 0, 0, 1)]
    probs, items = [], []
    for i, (N, K, s, fmt, group, bias, fp8) in enumerate(specs):
        p = synth.make_problem("mix", N, K, 16, s, seed=500 + 11 * i + M, group_size=group,
                               beta_std=0.002 if bias else 0.0, residual_fp8=bool(fp8))
        lay = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, group_size=group or K, fmt=fmt)
        lay.set_options((qt.QTEA_OPT_BIAS if bias else 0) | (qt.QTEA_OPT_RESIDUAL_FP8 if fp8 else 0))
        rv = dev(p.residual_vals) if fp8 else dev(p.residual_vals.view(np.int16), torch.float16)
        items.append(dict(x=dev(p.x[:M].view(np.int16), torch.float16), layout=lay,
                          row_scale=dev(scales(p, bias).view(np.int16), torch.float16),
                          col_scale=dev(p.v.view(np.int16), torch.float16), salient_idx=dev(p.salient_idx),
                          residual_vals=rv, residual_idx=dev(p.residual_idx)))
        probs.append((p, bias))
    ys = qt.qtea_gemv_grouped(items)
    torch.cuda.synchronize()
    for it in items:
        assert qt.qtea_device_status(it["layout"]) == 0
    for (p, bias), y in zip(probs, ys):
        y_ref, b = reference(p, bias, M=M)
        assert_within(y.cpu().numpy().astype(np.float64), y_ref, b, f"{p.N}x{p.K} M {M}")


@pytest.mark.parametrize("M", [1, 2, 4, 5])
def test_grouped_base3_calls(qt, M):
    """Eleven base-3 layouts in one grouped call (two launches of the staged fixed-point kernel at
    M <= 4, the general kernel at M = 5): ragged K against the 128-column blocks, groups of 128 or
    the whole row, with and without beta, FP8 or fp16 residual values, no residual with N not a
    multiple of 4, and a 2-bit layout in between that takes another kernel."""
    specs = [  # (N, K, s, fmt, group, bias, fp8)
        (256, 1024, 8, 1, 128, 1, 1), (64, 300, 4, 1, 0, 0, 0), (130, 700, 0, 1, 128, 1, 0),
        (512, 2048, 24, 1, 128, 0, 1), (36, 128, 4, 1, 0, 1, 1), (100, 257, 0, 1, 0, 0, 0),
        (64, 1024, 8, 0, 0, 1, 0), (128, 4096, 40, 1, 128, 1, 1), (260, 640, 12, 1, 128, 1, 0),
        (8, 1, 0, 1, 0, 0, 0), (1024, 512, 16, 1, 128, 1, 1), (68, 1920, 8, 1, 0, 1, 1)]
    probs, items = [], []
    for i, (N, K, s, fmt, group, bias, fp8) in enumerate(specs):
        p = synth.make_problem("b3", N, K, 16, s, seed=900 + 13 * i + M, group_size=group,
                               beta_std=0.002 if bias else 0.0, residual_fp8=bool(fp8))
        lay = qt.qtea_pack_layout(dev(p.T), n_salient=p.s, group_size=group or K, fmt=fmt)
        lay.set_options((qt.QTEA_OPT_BIAS if bias else 0) | (qt.QTEA_OPT_RESIDUAL_FP8 if fp8 else 0))
        rv = dev(p.residual_vals) if fp8 else dev(p.residual_vals.view(np.int16), torch.float16)
        items.append(dict(x=dev(p.x[:M].view(np.int16), torch.float16), layout=lay,
                          row_scale=dev(scales(p, bias).view(np.int16), torch.float16),
                          col_scale=dev(p.v.view(np.int16), torch.float16),
                          salient_idx=dev(p.salient_idx) if s else None, residual_vals=rv if s else None,
                          residual_idx=dev(p.residual_idx) if s else None))
        probs.append((p, bias))
    ys = qt.qtea_gemv_grouped(items)
    ys2 = qt.qtea_gemv_grouped(items)
    torch.cuda.synchronize()
    for it in items:
        assert qt.qtea_device_status(it["layout"]) == 0
    for (p, bias), y, y2 in zip(probs, ys, ys2):
        y_ref, b = reference(p, bias, M=M)
        assert_within(y.cpu().numpy().astype(np.float64), y_ref, b, f"{p.N}x{p.K} M {M}")
        assert torch.equal(y, y2), "repeated grouped calls differ"
