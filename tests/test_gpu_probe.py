"""The decode-rate diagnostic (qtea_probe_decode_rates): it runs and gives plausible rates.

It measures the instruction issue rates that decided the batch-1 decode (dp4a rather than
mma.sync with A built from the codes); the values are hardware facts, so the test checks only that
every rate is measured and positive, and that an MMA whose A operand changes every instruction is
no faster than one with constant operands.
"""
import pytest

torch = pytest.importorskip("torch")


@pytest.mark.gpu
def test_probe_decode_rates():
    import paper_2609_00224_gb300 as qt
    qt.load()
    r = qt.qtea_probe_decode_rates()
    assert set(r) == {"mma_m16n8k16_f16_constant", "mma_m16n8k16_f16_decoded_a", "mma_m16n8k32_e4m3_constant",
                      "mma_m16n8k32_e4m3_decoded_a", "dp4a"}
    assert all(0.25 < v < 1000 for v in r.values()), r
    assert r["mma_m16n8k16_f16_decoded_a"] >= 0.9 * r["mma_m16n8k16_f16_constant"], r
    assert r["mma_m16n8k32_e4m3_decoded_a"] >= 0.9 * r["mma_m16n8k32_e4m3_constant"], r
