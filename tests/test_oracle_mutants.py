"""Planted mistakes: each mutant of the oracle must fail at least one pin.

A copy of the oracle's C source gets one plausible error (a dropped term, a wrong sign,
index or bit order), is compiled into a temporary library, and is run through a compact
version of the pins in test_oracle.py. The real oracle must pass all of them; every
mutant must fail at least one, which shows the pins can see that kind of mistake.
"""
import os
import subprocess

import numpy as np
import pytest

import oracle
import synth
from test_oracle import residual_golden_case

F16 = np.float16
SRC = os.path.join(os.path.dirname(oracle.__file__), "qtea_oracle.c")


def f(bits):
    return np.asarray(bits, dtype=np.uint16).view(F16).astype(np.float64)


def dense(p, beta=None, g=None):
    N, K = p.T.shape
    g = K if g is None else g
    G = -(-K // g)
    cols = np.arange(K) // g
    a = f(p.alpha).reshape(N, G)[:, cols]
    b = 0 if beta is None else f(beta).reshape(N, G)[:, cols]
    W = a * f(p.v)[None] * p.T + b
    pos = synth.residual_positions(p.residual_idx, p.s)
    for q in range(N // 4 if p.s else 0):
        for c in range(p.s):
            W[4 * q + pos[q, c], p.salient_idx[c]] += f(p.residual_vals)[q, c]
    return W


def pin_failures(lib):
    """Names of the pins this oracle build fails."""
    fails = []

    def check(name, ok):
        if not ok:
            fails.append(name)

    # binary16 decoding of every pattern
    bits = np.arange(65536, dtype=np.uint32)
    ref = bits.astype(np.uint16).view(F16).astype(np.float64)
    got = np.array([lib.qo_half_to_double(int(b)) for b in bits])
    fin = np.isfinite(ref)
    check("half", np.array_equal(got[fin], ref[fin]))
    # brute force, one scale per row
    for (N, K, s, M) in [(8, 64, 8, 2), (64, 256, 8, 1)]:
        p = synth.make_problem("m", N, K, M, s, seed=N + K + s)
        try:
            y, b = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, lib=lib)
        except oracle.OracleError:
            check("dense", False)
            continue
        W = dense(p)
        x = f(p.x)
        check("dense", np.allclose(y, x @ W.T, rtol=1e-12, atol=1e-12))
        check("bound", np.allclose(b, np.abs(x[:, None, :] * W[None]).sum(-1), rtol=1e-12, atol=0))
    # brute force, group scales with bias (Eq. 10 in full)
    p = synth.make_problem("m", 8, 256, 2, 4, seed=77)
    p.alpha = synth.uniform_f16(1, 2, (8, 2), 0.01, 0.05)
    beta = synth.normal_f16(1, 9, (8, 2), 0.0, 0.01)
    y, _ = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx,
                       beta=beta, group_size=128, lib=lib)
    check("groups", np.allclose(y, f(p.x) @ dense(p, beta, 128).T, rtol=1e-12, atol=1e-13))
    # packing: known bytes and round trip
    T = np.zeros((1, 64), np.int8)
    T[0, :4] = [1, -1, 1, 0]
    check("pack2", int(oracle.pack(T, "2bit", lib=lib)[0]) == (2 | 0 << 2 | 2 << 4 | 1 << 6))
    T = np.zeros((1, 128), np.int8)
    T[0, :5] = [1, -1, 0, 0, 0]
    check("pack3", int(oracle.pack(T, "base3", lib=lib)[0]) == 119)
    # FP8 E4M3 residual values: the format's defining values, and a dense brute force with them
    table = {0x01: 2.0 ** -9, 0x07: 7 * 2.0 ** -9, 0x08: 2.0 ** -6, 0x38: 1.0, 0x7e: 448.0, 0xb8: -1.0}
    check("e4m3", all(lib.qo_e4m3_to_double(b) == v for b, v in table.items()) and
          np.isnan(lib.qo_e4m3_to_double(0x7f)))
    p = synth.make_problem("m", 8, 64, 2, 8, seed=91, residual_fp8=True)
    y, _ = oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, residual_fp8=True,
                       lib=lib)
    W = f(p.alpha) * f(p.v)[None] * p.T
    pos = synth.residual_positions(p.residual_idx, p.s)
    dec = {b: lib.qo_e4m3_to_double(int(b)) for b in range(256)} if "e4m3" not in fails else None
    if dec is not None:
        for q in range(2):
            for c in range(p.s):
                W[4 * q + pos[q, c], p.salient_idx[c]] += dec[int(p.residual_vals[q, c])]
        check("fp8_residual", np.allclose(y, f(p.x) @ W.T, rtol=1e-12, atol=1e-13))
    # residual positions from hand-written bytes (test_oracle.residual_golden_case)
    N, K, sal, ridx, R, rv, T, alpha, v = residual_golden_case()
    rows = [[1, 3, 0, 2, 2], [7, 6, 5, 4, 5]]
    ok = True
    for c, col in enumerate(sal):
        x = np.zeros((1, K), np.uint16)
        x[0, col] = synth.f16_from_double(1.0)
        try:
            y, _ = oracle.gemv(x, T, alpha, v, sal, rv, ridx, lib=lib)
        except oracle.OracleError:
            ok = False
            break
        want = np.zeros(N)
        want[rows[0][c]] += R[0, c]
        want[rows[1][c]] += R[1, c]
        ok = ok and np.array_equal(y[0], want)
    check("residual_golden", ok)
    # LUT symmetry and single-digit entries
    xs = np.array([0.3, -1.25, 2.0, 0.125, -0.5])
    lut = oracle.lut5(xs, lib=lib)
    check("lut", np.array_equal(lut, -lut[::-1]) and all(lut[121 + 3 ** d] == xs[d] for d in range(5)))
    # the salient bitmap of Sec. 3.5 from hand-written words
    try:
        idx = oracle.salient_from_bitmap(np.array([0x80000005, 0x81], np.uint32), 40, lib=lib)
        bm = oracle.salient_to_bitmap(np.array([0, 2, 31, 32, 39], np.int32), 40, lib=lib)
        check("bitmap", idx.tolist() == [0, 2, 31, 32, 39] and bm.tolist() == [0x80000005, 0x81])
    except oracle.OracleError:
        check("bitmap", False)
    return fails


MUTANTS = {
    "drop_residual_term": [("acc += residual_value(", "acc += 0.0 * residual_value(")],
    "e4m3_exponent_bias": [("expo - 10); /* (1 + frac/8)", "expo - 9); /* (1 + frac/8)")],
    "e4m3_subnormal_scale": [("ldexp((double)frac, -9);", "ldexp((double)frac, -10);")],
    "e4m3_nan_range": [("if (expo == 0xf && frac == 7) {", "if (expo == 0xf && frac >= 6) {")],
    "wrong_residual_row": [("== o % 4)\n          acc +=", "== (o + 1) % 4)\n          acc +=")],
    "ternary_sign_flip": [("tvx += (double)T[", "tvx -= (double)T[")],
    "rescale_index_shift": [("qo_half_to_double(v[j]) * xj", "qo_half_to_double(v[(j + 1) % K]) * xj")],
    "bias_times_rescaled_x": [("sx += xj;", "sx += xj * qo_half_to_double(v[j]);")],
    "alpha_first_group_only": [("double a = qo_half_to_double(alpha[(size_t)o * G + g]);\n        double b = beta ? qo_half_to_double(beta[(size_t)o * G + g]) : 0.0;\n        acc +=",
                                "double a = qo_half_to_double(alpha[(size_t)o * G]);\n        double b = beta ? qo_half_to_double(beta[(size_t)o * G + g]) : 0.0;\n        acc +=")],
    "transposed_codes": [("tvx += (double)T[(size_t)o * K + j]", "tvx += (double)T[((size_t)j * N + o) % ((size_t)N * K)]")],
    "bound_without_abs_w": [("fabs(qo_half_to_double(xm[j]) * w_row[j])", "fabs(qo_half_to_double(xm[j])) * w_row[j]")],
    "pack_msb_first": [("(uint8_t)(code << (2 * (k % 4)))", "(uint8_t)(code << (6 - 2 * (k % 4)))")],
    "half_exponent_bias": [("expo - 25", "expo - 24")],
    "half_subnormal_scale": [("ldexp((double)frac, -24)", "ldexp((double)frac, -23)")],
    "base3_digit_order": [("int value = 0, weight = 1;", "int value = 0, weight = 81;"), ("weight *= 3;", "weight /= 3;")],
    "lut_digit_offset": [("(double)(rest % 3 - 1) * xs[d]", "(double)(rest % 3) * xs[d]")],
    "residual_position_msb_first": [(">> (2 * (c % 4))) & 3;", ">> (6 - 2 * (c % 4))) & 3;")],
    "residual_position_byte_stride": [("ridx[(size_t)q * residual_stride(s) + c / 4]", "ridx[(size_t)q * (s / 4) + c / 4]")],
    "bitmap_msb_first": [("if ((bitmap[j / 32] >> (j % 32)) & 1u) {", "if ((bitmap[j / 32] >> (31 - j % 32)) & 1u) {"),
                         ("bitmap[idx[i] / 32] |= 1u << (idx[i] % 32);", "bitmap[idx[i] / 32] |= 1u << (31 - idx[i] % 32);")],
    "bitmap_word_stride": [("if ((bitmap[j / 32] >> (j % 32)) & 1u) {", "if ((bitmap[j / 31] >> (j % 32)) & 1u) {")],
}


@pytest.fixture(scope="module")
def mutant_dir(tmp_path_factory):
    return tmp_path_factory.mktemp("oracle_mutants")


def test_real_oracle_passes_every_pin():
    assert pin_failures(oracle.load()) == []


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, mutant_dir):
    src = open(SRC).read()
    for old, new in MUTANTS[name]:
        assert old in src, f"mutation anchor for {name} not found"
        src = src.replace(old, new)
    c_path = mutant_dir / f"{name}.c"
    so_path = mutant_dir / f"{name}.so"
    c_path.write_text(src)
    subprocess.check_call(["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-o", str(so_path), str(c_path), "-lm"])
    lib = oracle.load(str(so_path))
    assert pin_failures(lib), f"mutant {name} passed every pin"
