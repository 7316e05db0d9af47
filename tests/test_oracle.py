"""Pins of the CPU oracle against what the QTEA paper and plain mathematics fix.

Nothing here compares the oracle with itself: every expected value comes from a closed
form, a library routine (numpy's binary16 conversion, numpy matmul on a dense matrix), a
brute-force construction on tiny inputs, an invariant, or a number printed in the paper.
"""
import os

import numpy as np
import pytest

import oracle
import synth

F16 = np.float16


def h(a):
    """float values -> fp16 bit patterns (numpy's round-to-nearest-even)."""
    return np.asarray(a, dtype=np.float64).astype(F16).view(np.uint16)


def f(bits):
    return np.asarray(bits, dtype=np.uint16).view(F16).astype(np.float64)


def dense_weight(p, beta=None, group_size=None):
    """Brute force: materialise W^ [N][K] from the stored operands (Eq. 4 + residual)."""
    N, K = p.T.shape
    g = K if group_size is None else group_size
    G = -(-K // g)
    alpha = f(p.alpha).reshape(N, G)
    b = np.zeros((N, G)) if beta is None else f(beta).reshape(N, G)
    cols = np.arange(K) // g
    W = alpha[:, cols] * f(p.v)[None, :] * p.T.astype(np.float64) + b[:, cols]
    pos = synth.residual_positions(p.residual_idx, p.s)
    rv = f(p.residual_vals)
    for q in range(N // 4 if p.s else 0):
        for c in range(p.s):
            W[4 * q + pos[q, c], p.salient_idx[c]] += rv[q, c]
    return W


def run(p, **kw):
    return oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, **kw)


# ---------------------------------------------------------------- binary16 decoding

def test_half_to_double_matches_numpy_for_every_pattern():
    lib = oracle.load()
    bits = np.arange(65536, dtype=np.uint32)
    ref = bits.astype(np.uint16).view(F16).astype(np.float64)
    got = np.array([lib.qo_half_to_double(int(b)) for b in bits])
    finite = np.isfinite(ref)
    assert np.array_equal(got[finite], ref[finite])
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    assert np.array_equal(got[np.isinf(ref)], ref[np.isinf(ref)])


def test_generator_rounding_matches_numpy():
    rng = np.random.default_rng(7)
    vals = np.concatenate([
        rng.normal(0, 1, 4000), rng.normal(0, 0.02, 4000), rng.laplace(0, 0.01, 2000),
        np.array([0.0, -0.0, 65504.0, 65519.9, 65520.0, 1e-8, 2.0 ** -24, 2.0 ** -25, 3 * 2.0 ** -26,
                  2.0 ** -14, 2.0 ** -14 * (1 - 2.0 ** -11), 1 + 2.0 ** -11, 1 + 3 * 2.0 ** -11, -1e6]),
        (np.arange(-2048, 2048) + 0.5) * 2.0 ** -10,  # exact ties at every exponent near 1
    ])
    got = np.array([synth.f16_from_double(v) for v in vals], dtype=np.uint16)
    with np.errstate(over="ignore"):  # 65520 and -1e6 round to +-inf on purpose
        ref = vals.astype(F16).view(np.uint16)
    assert np.array_equal(got, ref)


# ---------------------------------------------------------------- brute force

@pytest.mark.parametrize("N,K,s,M", [(4, 8, 0, 1), (4, 8, 8, 3), (8, 64, 8, 1), (64, 128, 8, 3),
                                     (64, 256, 0, 3), (64, 256, 8, 1), (8, 100, 4, 2)])
def test_matches_dense_dequantize_then_matmul(N, K, s, M):
    p = synth.make_problem("t", N, K, M, s, seed=N * 1000 + K * 10 + s + M)
    y, bound = run(p)
    W = dense_weight(p)
    x = f(p.x)
    y_ref = x @ W.T
    b_ref = np.abs(x[:, None, :] * W[None, :, :]).sum(-1)
    assert np.allclose(y, y_ref, rtol=1e-12, atol=1e-12 * np.abs(b_ref).max())
    assert np.allclose(bound, b_ref, rtol=1e-12, atol=0)


@pytest.mark.parametrize("K,g", [(256, 128), (300, 128), (64, 16)])
def test_group_scales_and_bias_match_dense(K, g):
    """Eq. 10 in full: per-(row, group) alpha and beta, beta multiplying sum(x) only."""
    N, M, s = 8, 2, 4
    p = synth.make_problem("t", N, K, M, s, seed=K + g)
    G = -(-K // g)
    p.alpha = synth.uniform_f16(11, 2, (N, G), 0.01, 0.05)
    beta = synth.normal_f16(11, 9, (N, G), 0.0, 0.01)
    y, _ = run(p, beta=beta, group_size=g)
    W = dense_weight(p, beta=beta, group_size=g)
    assert np.allclose(y, f(p.x) @ W.T, rtol=1e-12, atol=1e-13)


# ---------------------------------------------------------------- FP8 E4M3 residual values

def _golden_e4m3():
    path = os.path.join(os.path.dirname(__file__), "golden", "e4m3_values.txt")
    rows = []
    for line in open(path):
        line = line.strip()
        if line and not line.startswith("#"):
            b, v = line.split()
            rows.append((int(b, 16), float(v)))
    return rows


def test_e4m3_decode_matches_the_format_table():
    """Values the FP8 E4M3 definition fixes (tests/golden/e4m3_values.txt, OFP8 Table 1)."""
    for b, v in _golden_e4m3():
        got = oracle.e4m3_to_double(b)
        if np.isnan(v):
            assert np.isnan(got), hex(b)
        else:
            assert got == v and np.signbit(got) == np.signbit(v), (hex(b), got, v)


def test_e4m3_values_are_exact_binary16_and_ordered():
    """Every finite E4M3 value is a binary16 value (numpy round trip is exact); the positive
    codes 0x00..0x7e are strictly increasing and the negative codes mirror them."""
    vals = np.array([oracle.e4m3_to_double(b) for b in range(256)])
    finite = ~np.isnan(vals)
    assert finite.sum() == 254
    assert np.array_equal(vals[finite].astype(F16).astype(np.float64), vals[finite])
    pos = vals[:0x7f]
    assert np.all(np.diff(pos) > 0)
    assert np.array_equal(vals[0x80:0xff], -pos)


def test_fp8_residual_equals_the_same_values_in_fp16():
    """The FP8 path adds the decoded value and nothing else: converting each E4M3 value to its
    (exactly equal) binary16 pattern gives the same y and bound."""
    N, K, M, s = 16, 256, 2, 24
    p = synth.make_problem("t", N, K, M, s, seed=77, residual_fp8=True)
    y8, b8 = run(p, residual_fp8=True)
    as16 = h([oracle.e4m3_to_double(b) for b in p.residual_vals.ravel()]).reshape(p.residual_vals.shape)
    y16, b16 = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, as16, p.residual_idx)
    assert np.array_equal(y8, y16) and np.array_equal(b8, b16)


def test_paper_storage_matches_dense():
    """The paper's own storage end to end: alpha and beta per (row, 128-column group), FP8 E4M3
    residual values; brute-force dense W^ (E4M3 decoded by the pinned routine) times x."""
    p = synth.paper_problem("tiny_1024", 0)
    p.T, p.x = p.T[:64, :300], p.x[:, :300]  # a ragged last group
    N, K = p.T.shape
    G = -(-K // 128)
    p.alpha, p.beta = p.alpha[:N, :G], p.beta[:N, :G]
    p.v = p.v[:K]
    keep = p.salient_idx < K
    p.salient_idx, p.s = p.salient_idx[keep], int(keep.sum())
    cols = np.flatnonzero(keep)
    p.residual_vals = np.ascontiguousarray(p.residual_vals[:N // 4][:, cols])
    pos = synth.residual_positions(p.residual_idx[:N // 4], 32)[:, cols]
    packed = np.zeros((N // 4, -(-p.s // 4)), np.uint8)
    for c in range(p.s):
        packed[:, c // 4] |= (pos[:, c] << (2 * (c % 4))).astype(np.uint8)
    p.residual_idx = packed
    y, _ = run(p, beta=p.beta, group_size=128, residual_fp8=True)
    alpha, beta = f(p.alpha), f(p.beta)
    g = np.arange(K) // 128
    W = alpha[:, g] * f(p.v)[None, :] * p.T + beta[:, g]
    for q in range(N // 4):
        for c in range(p.s):
            W[4 * q + pos[q, c], p.salient_idx[c]] += oracle.e4m3_to_double(p.residual_vals[q, c])
    assert np.allclose(y, f(p.x) @ W.T, rtol=1e-12, atol=1e-13)


def test_generator_e4m3_rounding_is_nearest_even():
    """The input generator's FP8 rounding against brute force over every finite E4M3 value
    (nearest, ties to the even code), with saturation at 448."""
    codes = [b for b in range(0x7f)]
    vals = np.array([oracle.e4m3_to_double(b) for b in codes])
    rng = np.random.default_rng(3)
    xs = np.concatenate([rng.normal(0, 0.02, 2000), rng.normal(0, 30, 2000), (vals[:-1] + vals[1:]) / 2,
                         vals, [500.0, 1e-12, 2.0 ** -10, 3 * 2.0 ** -11]])
    for x in xs:
        a = abs(x)
        if a >= 448:
            want = 0x7e
        else:
            d = np.abs(vals - a)
            cand = np.flatnonzero(d == d.min())
            want = int(cand[0]) if len(cand) == 1 else int([c for c in cand if c % 2 == 0][0])
        want |= 0x80 if np.signbit(x) else 0
        assert synth.e4m3_from_double(x) == want, (x, hex(want))


# ---------------------------------------------------------------- closed forms

def test_unit_vector_extracts_a_column():
    p = synth.make_problem("t", 16, 64, 1, 8, seed=5)
    W = dense_weight(p)
    for k in [0, 7, int(p.salient_idx[0]), int(p.salient_idx[-1]), 63]:
        p.x = h(np.eye(64)[k:k + 1])
        y, _ = run(p)
        # y[o] = W^[o][k] = alpha_o v_k T_ok (+ R where column k is salient)
        expect = f(p.alpha)[:, 0] * f(p.v)[k] * p.T[:, k]
        if k in set(p.salient_idx.tolist()):
            c = int(np.searchsorted(p.salient_idx, k))
            pos = synth.residual_positions(p.residual_idx, p.s)[:, c]
            expect = expect + np.where(np.arange(16) % 4 == np.repeat(pos, 4), np.repeat(f(p.residual_vals)[:, c], 4), 0)
        assert np.array_equal(y[0], expect)
        assert np.array_equal(y[0], W[:, k])


@pytest.mark.parametrize("t", [1, -1])
def test_constant_codes_give_plus_minus_sum_x(t):
    N, K = 8, 96
    p = synth.make_problem("t", N, K, 2, 0, seed=3)
    p.T[:] = t
    p.alpha[:] = h(1.0)
    p.v[:] = h(1.0)
    y, _ = run(p)
    sx = f(p.x).sum(axis=1)
    assert np.allclose(y, t * sx[:, None], rtol=0, atol=1e-12)


def test_signed_sum_by_counting():
    p = synth.make_problem("t", 12, 200, 1, 0, seed=4)
    p.alpha[:] = h(1.0)
    p.v[:] = h(1.0)
    y, _ = run(p)
    x = f(p.x)[0]
    expect = [(x[p.T[o] == 1]).sum() - (x[p.T[o] == -1]).sum() for o in range(12)]
    assert np.allclose(y[0], expect, rtol=0, atol=1e-12)


def test_zero_residual_is_pure_ternary():
    p = synth.make_problem("t", 32, 128, 2, 16, seed=6)
    p.residual_vals[:] = 0
    y, _ = run(p)
    y0, _ = oracle.gemv(p.x, p.T, p.alpha, p.v)
    assert np.array_equal(y, y0)
    expect = (f(p.x) * f(p.v)[None]) @ p.T.T.astype(np.float64) * f(p.alpha)[:, 0][None]
    assert np.allclose(y, expect, rtol=1e-13, atol=1e-13)


def test_one_salient_column_closed_form():
    N, K, jstar = 16, 64, 37
    p = synth.make_problem("t", N, K, 1, 1, seed=8)
    p.T[:] = 0
    p.salient_idx = np.array([jstar], np.int32)
    y, _ = run(p)
    pos = synth.residual_positions(p.residual_idx, 1)[:, 0]
    r = f(p.residual_vals)[:, 0]
    xj = f(p.x)[0, jstar]
    expect = np.array([r[o // 4] * xj if pos[o // 4] == o % 4 else 0.0 for o in range(N)])
    assert np.array_equal(y[0], expect)
    assert np.count_nonzero(expect) <= N // 4  # exactly one entry per group of four rows


def test_linearity_and_batch_independence():
    p = synth.make_problem("t", 16, 64, 3, 8, seed=9)
    rng = np.random.default_rng(0)
    x1 = rng.integers(-8, 9, (1, 64)).astype(np.float64)
    x2 = rng.integers(-8, 9, (1, 64)).astype(np.float64)
    ys = []
    for xv in (x1, x2, 2 * x1 - x2):
        p.x = h(xv)
        ys.append(run(p)[0][0])
    assert np.allclose(ys[2], 2 * ys[0] - ys[1], rtol=1e-12, atol=1e-12)
    p = synth.make_problem("t", 16, 64, 3, 8, seed=10)
    y, b = run(p)
    for m in range(3):
        ym, bm = oracle.gemv(p.x[m:m + 1], p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx)
        assert np.array_equal(ym[0], y[m]) and np.array_equal(bm[0], b[m])


def test_row_subset_matches_full():
    p = synth.make_problem("t", 64, 256, 2, 8, seed=12)
    y, b = run(p)
    rows = np.array([63, 0, 17, 4, 5], np.int32)
    ys, bs = run(p, rows=rows)
    assert np.array_equal(ys, y[:, rows]) and np.array_equal(bs, b[:, rows])


def test_bound_properties():
    p = synth.make_problem("t", 32, 128, 2, 8, seed=13)
    y, b = run(p)
    assert np.all(b >= np.abs(y) - 1e-15)
    p.x = (p.x ^ np.uint16(0x8000))  # negate x: y flips sign, bound unchanged
    y2, b2 = run(p)
    assert np.array_equal(y2, -y) and np.array_equal(b2, b)


def test_rejects_bad_inputs():
    p = synth.make_problem("t", 8, 16, 1, 4, seed=14)
    T = p.T.copy()
    T[3, 5] = 2
    with pytest.raises(oracle.OracleError):
        oracle.gemv(p.x, T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx)
    sal = p.salient_idx.copy()
    sal[1] = sal[0]
    with pytest.raises(oracle.OracleError):
        oracle.gemv(p.x, p.T, p.alpha, p.v, sal, p.residual_vals, p.residual_idx)


# ---------------------------------------------------------------- packed layouts

def residual_golden_case():
    """Two groups of four rows, five salient columns, no ternary part: y = x * R placed by the
    positions. The position bytes are written by hand from the layout rule (entry c of group q at
    bits 2 (c % 4) of byte q * ceil(s/4) + c / 4): group 0 positions [1, 3, 0, 2 | 2] are bytes
    0x8D (1 + 3*4 + 0*16 + 2*64) and 0x02; group 1 positions [3, 2, 1, 0 | 1] are 0x1B and 0x01."""
    N, K, s = 8, 8, 5
    sal = np.array([1, 2, 4, 6, 7], np.int32)
    ridx = np.array([[0x8D, 0x02], [0x1B, 0x01]], np.uint8)
    one = synth.f16_from_double(1.0)
    R = np.array([[0.5, 0.25, -1.0, 2.0, 0.125], [-0.5, 4.0, 0.75, -2.0, 1.5]])
    rv = np.array([[synth.f16_from_double(r) for r in row] for row in R], np.uint16)
    T = np.zeros((N, K), np.int8)
    alpha = np.full((N, 1), one, np.uint16)
    v = np.full(K, one, np.uint16)
    return N, K, sal, ridx, R, rv, T, alpha, v


def test_residual_positions_hand_written_bytes():
    N, K, sal, ridx, R, rv, T, alpha, v = residual_golden_case()
    # expected rows of every entry, read off the hand-written positions above
    rows = {(0, 0): 1, (0, 1): 3, (0, 2): 0, (0, 3): 2, (0, 4): 2,
            (1, 0): 7, (1, 1): 6, (1, 2): 5, (1, 3): 4, (1, 4): 5}
    for c, col in enumerate(sal):
        x = np.zeros((1, K), np.uint16)
        x[0, col] = synth.f16_from_double(1.0)
        y, _ = oracle.gemv(x, T, alpha, v, sal, rv, ridx)
        want = np.zeros(N)
        want[rows[(0, c)]] += R[0, c]
        want[rows[(1, c)]] += R[1, c]
        assert np.array_equal(y[0], want), (c, y[0], want)


def test_pack_2bit_known_bytes_and_padding():
    for t, byte in [(-1, 0x00), (0, 0x55), (1, 0xAA)]:
        T = np.full((3, 8), t, np.int8)
        packed = oracle.pack(T, "2bit").reshape(3, 16)  # K_pad = 64 -> 16 bytes per row
        assert np.all(packed[:, :2] == byte)
        assert np.all(packed[:, 2:] == 0x55)  # pad columns hold code 1 (T = 0)
    T = np.zeros((1, 64), np.int8)
    T[0, 0], T[0, 1], T[0, 2], T[0, 3], T[0, 63] = 1, -1, 1, 0, -1
    packed = oracle.pack(T, "2bit")
    assert packed[0] == (2 | 0 << 2 | 2 << 4 | 1 << 6)  # least significant code first
    assert packed[15] == (1 | 1 << 2 | 1 << 4 | 0 << 6)
    assert oracle.packed_bytes(4096, 4096) == 4096 * 1024
    assert oracle.packed_bytes(3, 65) == 3 * 32


def test_pack_base3_known_bytes():
    # five ternary digits per byte (3^5 = 243 < 256), 26 bytes per 128 columns, 2 pad digits
    for t, full, last in [(-1, 0, 0 + 0 + 0 + 27 + 81), (1, 242, 2 + 6 + 18 + 27 + 81), (0, 121, 121)]:
        packed = oracle.pack(np.full((2, 128), t, np.int8), "base3").reshape(2, 26)
        assert np.all(packed[:, :25] == full) and np.all(packed[:, 25] == last)
    T = np.zeros((1, 128), np.int8)
    T[0, :5] = [1, -1, 0, 0, 0]  # digits 2, 0, 1, 1, 1 -> 2 + 0*3 + 9 + 27 + 81
    assert oracle.pack(T, "base3")[0] == 119
    # storage ratio vs fp16 (Appendix A: "about 9.85x smaller"): 128 * 2 bytes / 26 bytes
    assert round(128 * 2 / 26, 2) == 9.85
    assert oracle.packed_bytes(4, 129, "base3") == 4 * 2 * 26


@pytest.mark.parametrize("fmt", ["2bit", "base3"])
@pytest.mark.parametrize("N,K", [(1, 1), (5, 63), (4, 64), (7, 130), (16, 640)])
def test_pack_roundtrip(fmt, N, K):
    T = synth.codes(N * 31 + K, 1, (N, K), 0.3, 0.4)
    assert np.array_equal(oracle.unpack(oracle.pack(T, fmt), N, K, fmt), T)


def test_unpack_rejects_illegal_code():
    packed = oracle.pack(np.zeros((1, 64), np.int8))
    packed[0] |= 0x03
    with pytest.raises(oracle.OracleError):
        oracle.unpack(packed, 1, 64)


# ---------------------------------------------------------------- LUT (Sec. 3.5)

def test_lut_sign_symmetry_and_zero_pattern():
    xs = np.array([0.3, -1.25, 2.0, 0.125, -0.5])
    lut = oracle.lut5(xs)
    # pattern -p has digits 2 - d, i.e. code 242 - c; its dot product is the negative
    assert np.array_equal(lut, -lut[::-1])
    assert lut[121] == 0.0
    assert lut[242] == xs.sum() and lut[0] == -xs.sum()
    for d in range(5):  # a single +1 digit (others 0) picks out one activation
        code = 121 + 3 ** d
        assert lut[code] == xs[d]


# ---------------------------------------------------------------- paper arithmetic (Appendix A)

def _asic_table():
    rows = []
    path = os.path.join(os.path.dirname(__file__), "golden", "asic_latency_table.txt")
    for line in open(path):
        if line.strip() and not line.startswith("#"):
            rows.append([float(v) for v in line.split()])
    return rows


def test_asic_latency_model_reproduces_paper_table():
    rows = _asic_table()
    assert len(rows) == 4
    speedups = []
    for K, N, fp16_us, qtea_us, _, _ in rows:
        t_tern, t_dense = oracle.asic_latency_us(int(K), int(N))
        assert round(t_tern, 2) == qtea_us
        assert round(t_dense, 2) == fp16_us
        speedups.append(t_dense / t_tern)
    assert round(float(np.mean(speedups)), 2) == 3.83
    energy_cut = np.mean([1 - r[5] / r[4] for r in rows])
    assert round(100 * float(energy_cut), 1) == 69.4


# ---------------------------------------------------------------- generated inputs

def test_generated_inputs_invariants():
    p = synth.workload_problem("llama3_8b_layer", 1)  # k_proj 1024 x 4096
    assert p.T.dtype == np.int8 and set(np.unique(p.T).tolist()) <= {-1, 0, 1}
    n = p.T.size
    for val, prob in [(-1, 0.3), (0, 0.4), (1, 0.3)]:
        cnt = np.count_nonzero(p.T == val)
        assert abs(cnt - n * prob) < 4 * np.sqrt(n * prob * (1 - prob))
    assert p.s == 120 and np.all(np.diff(p.salient_idx) > 0) and 0 <= p.salient_idx[0] and p.salient_idx[-1] < p.K
    pos = synth.residual_positions(p.residual_idx, p.s)
    assert pos.shape == (p.N // 4, p.s) and pos.max() <= 3  # one position per (group, column)
    a = f(p.alpha)
    assert a.min() >= 0.01 - 1e-5 and a.max() <= 0.05 + 1e-5
    v = f(p.v)
    assert v.min() >= 0.8 - 1e-3 and v.max() <= 1.2 + 1e-3
    x = f(p.x)
    assert abs(x.mean()) < 0.1 and abs(x.std() - 1) < 0.05
    r = f(p.residual_vals)
    assert abs(r.std() - 0.02) < 0.002
    assert [synth.salient_count(K) for K in (4096, 5120, 8192, 14336, 17408, 28672)] == [120, 152, 248, 432, 520, 864]


def test_generator_is_deterministic_and_thread_independent():
    a = synth.codes(123, 1, (3000, 700), 0.3, 0.4)  # > 2^20 elements: multithreaded
    b = synth.codes(123, 1, (3000, 700), 0.3, 0.4)
    c = synth.codes(123, 1, (10, 700), 0.3, 0.4)    # single thread, same stream prefix
    assert np.array_equal(a, b) and np.array_equal(a[:10], c)


# ---------------------------------------------------------------- salient bitmap (Sec. 3.5)

def test_salient_bitmap_known_words():
    """Sec. 3.5 stores the salient set as a bitmap over input columns. Hand-worked: word 0 =
    0x80000005 marks columns 0, 2 and 31; word 1 = 0x81 marks columns 32 + 0 and 32 + 7."""
    words = np.array([0x80000005, 0x81], np.uint32)
    assert oracle.salient_from_bitmap(words, 40).tolist() == [0, 2, 31, 32, 39]
    assert oracle.salient_to_bitmap(np.array([0, 2, 31, 32, 39], np.int32), 40).tolist() == [0x80000005, 0x81]


def test_salient_bitmap_ignores_bits_past_k():
    # K = 35: only columns 32, 33, 34 of word 1 exist
    assert oracle.salient_from_bitmap(np.array([0, 0xFFFFFFFF], np.uint32), 35).tolist() == [32, 33, 34]
    assert oracle.salient_from_bitmap(np.zeros(0, np.uint32), 0).tolist() == []


def test_salient_bitmap_round_trip_and_rejects_bad_lists():
    rng = np.random.default_rng(5)
    for K in (1, 31, 32, 33, 1000, 4096):
        idx = np.sort(rng.choice(K, size=min(K, max(1, K // 10)), replace=False)).astype(np.int32)
        bm = oracle.salient_to_bitmap(idx, K)
        assert bm.size == (K + 31) // 32
        assert np.array_equal(oracle.salient_from_bitmap(bm, K), idx)
        # popcount equals the list length (no bit set twice, none lost)
        assert sum(bin(int(w)).count("1") for w in bm) == idx.size
    for bad in ([3, 3], [5, 2], [-1], [40]):
        with pytest.raises(oracle.OracleError):
            oracle.salient_to_bitmap(np.array(bad, np.int32), 40)
