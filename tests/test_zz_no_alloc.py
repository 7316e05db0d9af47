"""qtea_gemv_m1_static, the allocation-free batch-1 entry point, against qtea_gemv.

The file name sorts last so that the GPU tests here also run after every other test has used the
library in the same process. Each case calls the static entry twice in a row: the second call
checks that the first left the static scratch's split-tile partial rows at zero (a row left set
would be added to the second call's sums), and qtea_gemv_m1_static_status confirms the scratch
is back in its start state.
Pass rule: the static entry runs the same kernel on the same grid as qtea_gemv, so its y equals
qtea_gemv's bit for bit, on both calls; both are within 1e-4 * sum_j |x_j * W^[o][j]| + 1e-6 of the
oracle's y. The calls allocate nothing: the device's free memory does not change across them.
"""
import ctypes

import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")

REL, ABS = 1e-4, 1e-6


@pytest.fixture(scope="module")
def qt():
    import paper_2609_00224_gb300 as m
    m.load()
    return m


def test_static_entry_host_checks_need_no_gpu(qt):
    lib = qt.load()
    call = lib.qtea_gemv_m1_static
    # sizes beyond the static scratch are refused before any CUDA call
    assert call(None, None, 131076, 64, 0, None, None, None, None, None, None, None) == qt.QTEA_ERR_SCRATCH_LIMIT
    assert "static scratch" in qt.status_string(qt.QTEA_ERR_SCRATCH_LIMIT)
    assert call(None, None, -1, 64, 0, None, None, None, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG
    assert call(None, None, 6, 64, 4, None, None, None, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG  # N % 4
    assert call(None, None, 4, 64, 65, None, None, None, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG  # s > K
    assert call(None, None, 4, 64, 0, None, None, None, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG  # no y
    assert call(None, None, 0, 64, 0, None, None, None, None, None, None, None) == qt.QTEA_OK  # empty


def _dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.cuda()


CASES = [
    ("tiny 1024x1024", lambda: synth.workload_problem("tiny_1024", 0)),
    ("ragged 1000x1000", lambda: synth.make_problem("r", 1000, 1000, 1, 24, seed=11)),
    ("llama3-8b down_proj 4096x14336", lambda: synth.workload_problem("llama3_8b_layer", 6)),
    ("llama3-8b gate_proj 14336x4096", lambda: synth.workload_problem("llama3_8b_layer", 4)),
    ("no residual 2048x3000", lambda: synth.make_problem("n", 2048, 3000, 1, 0, seed=12)),
]


@pytest.mark.gpu
@pytest.mark.parametrize("name,make", CASES, ids=[c[0] for c in CASES])
def test_static_entry_matches_qtea_gemv(qt, name, make):
    p = make()
    T = _dev(p.T)
    layout = qt.qtea_pack_layout(T, n_salient=p.s)
    # the static entry runs the stream-K batch-1 kernel: qtea_gemv pinned to the same kernel agrees bitwise
    layout.set_options(qt.QTEA_OPT_STREAM_K)
    packed = qt.packed_bytes(layout).clone()  # caller-owned copy of the 2-bit layout
    x = _dev(p.x.view(np.int16), torch.float16)
    alpha = _dev(p.alpha.reshape(-1).view(np.int16), torch.float16)
    v = _dev(p.v.view(np.int16), torch.float16)
    sal = _dev(p.salient_idx) if p.s else None
    rv = _dev(p.residual_vals.view(np.int16), torch.float16) if p.s else None
    ri = _dev(p.residual_idx) if p.s else None

    y_api = qt.qtea_gemv(x, layout, alpha, v, sal, rv, ri)
    torch.cuda.synchronize()
    assert qt.qtea_device_status(layout) == 0

    def ptr(t):
        return None if t is None else t.data_ptr()

    lib = qt.load()
    stream = torch.cuda.current_stream().cuda_stream
    ys = [torch.full((1, p.N), float("nan"), dtype=torch.float32, device="cuda") for _ in range(2)]
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for y in ys:
        rc = lib.qtea_gemv_m1_static(ptr(x), ptr(packed), p.N, p.K, p.s, ptr(alpha), ptr(v), ptr(sal), ptr(rv),
                                     ptr(ri), ptr(y), ctypes.c_void_p(stream))
        assert rc == qt.QTEA_OK, qt.status_string(rc)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0, "the static entry changed the device's free memory"
    assert lib.qtea_gemv_m1_static_status(0, ctypes.c_void_p(stream)) == qt.QTEA_OK

    y_ref, bound = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx)
    lim = REL * bound.reshape(-1) + ABS
    ya = y_api.cpu().numpy().astype(np.float64).reshape(-1)
    assert np.all(np.abs(ya - y_ref.reshape(-1)) <= lim)
    for k, y in enumerate(ys):
        yk = y.cpu().numpy().astype(np.float64).reshape(-1)
        assert np.all(np.isfinite(yk)), f"call {k + 1}: unwritten outputs"
        assert torch.equal(y, y_api), f"call {k + 1}: differs from qtea_gemv"
        assert np.all(np.abs(yk - y_ref.reshape(-1)) <= lim)


@pytest.mark.gpu
def test_static_entry_sees_codes_written_just_before_it(qt):
    """The caller rewrites its packed codes with a kernel on the same stream right before the call
    (programmatic dependent launch must not let the call read them early): y follows the new codes."""
    qt_ = qt
    p = synth.workload_problem("llama3_8b_layer", 4)  # gate_proj 14336 x 4096
    q = synth.make_problem("other codes", p.N, p.K, 1, p.s, seed=77)
    lay_p = qt_.qtea_pack_layout(_dev(p.T), n_salient=p.s)
    lay_q = qt_.qtea_pack_layout(_dev(q.T), n_salient=p.s)
    lay_q.set_options(qt_.QTEA_OPT_STREAM_K)  # the static entry's kernel, for a bitwise comparison
    codes_q = qt_.packed_bytes(lay_q).clone()
    packed = qt_.packed_bytes(lay_p).clone()
    x = _dev(p.x.view(np.int16), torch.float16)
    alpha = _dev(p.alpha.reshape(-1).view(np.int16), torch.float16)
    v = _dev(p.v.view(np.int16), torch.float16)
    sal, rv, ri = _dev(p.salient_idx), _dev(p.residual_vals.view(np.int16), torch.float16), _dev(p.residual_idx)
    y_q = qt_.qtea_gemv(x, lay_q, alpha, v, sal, rv, ri)  # q's codes with p's other operands
    y = torch.empty((1, p.N), dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    lib = qt_.load()
    stream = torch.cuda.current_stream()
    for _ in range(3):
        packed.copy_(codes_q)  # a kernel on the stream writes the codes ...
        rc = lib.qtea_gemv_m1_static(x.data_ptr(), packed.data_ptr(), p.N, p.K, p.s, alpha.data_ptr(), v.data_ptr(),
                                     sal.data_ptr(), rv.data_ptr(), ri.data_ptr(), y.data_ptr(),
                                     ctypes.c_void_p(stream.cuda_stream))  # ... and the call follows it
        assert rc == qt_.QTEA_OK
        torch.cuda.synchronize()
        assert torch.equal(y, y_q)
        packed.copy_(qt_.packed_bytes(lay_p))  # back to p's codes for the next round
        torch.cuda.synchronize()
    assert lib.qtea_gemv_m1_static_status(0, ctypes.c_void_p(stream.cuda_stream)) == qt_.QTEA_OK
