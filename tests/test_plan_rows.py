"""The batch-1 dispatch rule, checked on the host (no device): which calls take the row-resident
launch, with how many CTAs, how many rows per CTA, whether the launch is wide, and how many lanes a
row gets (qtea_rows_plan_shapes, the shape-level core of the plan qtea_gemv_grouped applies).

Pins: the launches the GPU captures recorded for the Llama3-8B calls (the q, k, v group on 304 CTAs
of 24 rows at most with CTAs of different lanes per row, o_proj on 152 CTAs of one lane per row,
k_proj on 128 CTAs of 8 rows), the measured limits (gate_proj and down_proj on the stream-K launch;
the Qwen3-14B and Llama3-70B k_proj on wide launches), and invariants every plan keeps.
"""
import random

import pytest

import paper_2609_00224_gb300 as qt

SM, OPTIN = 152, 232448  # GB300: SMs, opt-in shared memory per block
L8 = dict(q=(4096, 4096, 120), k=(1024, 4096, 120), v=(1024, 4096, 120), o=(4096, 4096, 120),
          gate=(14336, 4096, 120), up=(14336, 4096, 120), down=(4096, 14336, 432))


def plan(shapes, sm=SM, optin=OPTIN):
    return qt.qtea_rows_plan_shapes(shapes, sm, optin)


def test_llama3_8b_calls():
    p = plan([L8["q"], L8["k"], L8["v"]])
    assert (p["grid"], p["rows_cap"], p["wide"], p["kparts"]) == (304, 24, 0, 0)
    assert p["ctas"][1] == p["ctas"][2] and sum(p["ctas"]) == 304
    p = plan([L8["o"]])
    assert (p["grid"], p["rows_cap"], p["wide"], p["kparts"]) == (152, 32, 0, 1)
    assert plan([L8["q"]])["grid"] == 152
    p = plan([L8["k"]])
    assert (p["grid"], p["rows_cap"], p["wide"], p["kparts"]) == (128, 8, 0, 4)
    for name in ("gate", "up", "down"):
        assert plan([L8[name]]) is None, name
    assert plan(list(L8.values())) is None


def test_wide_launches_and_limits():
    for shape in ((1024, 5120, 152), (1024, 8192, 248)):  # Qwen3-14B and Llama3-70B k_proj
        p = plan([shape])
        assert (p["grid"], p["rows_cap"], p["wide"], p["kparts"]) == (128, 8, 1, 4)
    assert plan([(1024, 4096, 300)])["wide"] == 1         # more than 256 salient columns
    assert plan([(1024, 4096, 256)])["wide"] == 0
    assert plan([(64, 8192, 512)])["wide"] == 1           # 16 chunks, 512 salient columns
    assert plan([(64, 8193, 8)]) is None                  # 17 chunks
    assert plan([(64, 4096, 513)]) is None                # 513 salient columns
    rows40 = 8 * (4 * SM + 1)                             # 40 rows per CTA with one CTA per SM
    narrow = plan([(rows40, 4096, 8)])
    assert narrow["grid"] == 2 * SM and narrow["rows_cap"] == 24 and narrow["wide"] == 0
    assert plan([(rows40, 4608, 8)]) is None              # wide: never two CTAs per SM
    p = plan([(512, 8192, 64), (256, 4096, 300), (128, 2048, 16)])
    assert (p["grid"], p["rows_cap"], p["wide"]) == (112, 8, 1) and p["ctas"] == [64, 32, 16]


def test_shared_memory_and_sm_count_bound_the_plan():
    assert plan([L8["q"], L8["k"], L8["v"]], optin=40 * 1024) is None  # needs 41,280 bytes
    assert plan([L8["o"]], sm=132)["grid"] == 132                      # 4096 rows: 32 per CTA on 128 CTAs
    p = plan([L8["o"]], sm=100)                                        # 48 rows on one CTA per SM: two
    assert (p["grid"], p["rows_cap"]) == (200, 24)
    assert plan([(64, 512, 0)] * 3, sm=2) is None                       # more problems than SMs


def test_plan_invariants_over_random_shape_sets():
    rng = random.Random(20260)
    fits = 0
    for _ in range(3000):
        n = rng.randint(1, 8)
        shapes = []
        for _ in range(n):
            K = rng.choice([64, 512, 1000, 2048, 4096, 4608, 5120, 8192, 8200, 14336])
            s = rng.choice([0, 8, 120, 256, 300, 512, 600])
            s = min(s, K)
            N = 4 * rng.randint(1, 1600)
            shapes.append((N, K, s))
        sm = rng.choice([16, 132, 152])
        p = plan(shapes, sm=sm)
        if p is None:
            continue
        fits += 1
        wide = any(-(-K // 512) > 8 or s > 256 for _, K, s in shapes)
        assert p["wide"] == int(wide)
        assert all(-(-K // 512) <= 16 and s <= 512 for _, K, s in shapes)
        assert sum(p["ctas"]) == p["grid"] <= (1 if wide else 2) * sm
        assert all(1 <= c <= -(-N // 8) for c, (N, _, _) in zip(p["ctas"], shapes))
        rows = max(-(-(-(-N // 8)) // c) * 8 for c, (N, _, _) in zip(p["ctas"], shapes))
        assert rows == p["rows_cap"] <= 32
        assert p["kparts"] in (0, 1, 2, 4)
    assert fits >= 150  # enough fitting plans for the invariants to mean something


def test_invalid_arguments():
    for shapes in ([(0, 512, 0)], [(4, 0, 0)], [(4, 64, 65)], [(6, 64, 4)], [(4, 70000, 0)]):
        with pytest.raises(qt.QteaError):
            plan(shapes)
    with pytest.raises(qt.QteaError):
        plan([(4, 64, 0)] * 9)
    with pytest.raises(qt.QteaError):
        plan([(4, 64, 0)], sm=0)
    with pytest.raises(qt.QteaError):
        plan([])
