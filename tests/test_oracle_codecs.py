"""Pins of the oracle's format decoders (OCP OFP8 E4M3, OCP MX E2M1, bf16)."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from tests import indep


def test_e4m3_all_256_codes_match_torch():
    ref = indep.e4m3_torch(np.arange(256, dtype=np.uint8))
    for c in range(256):
        v = oracle.e4m3(c)
        if c in (0x7F, 0xFF):
            assert math.isnan(v) and math.isnan(ref[c])
        else:
            assert v == ref[c], hex(c)
            assert math.copysign(1.0, v) == math.copysign(1.0, ref[c]), hex(c)


def test_e4m3_spec_table():
    for code, val in indep.read_table("e4m3_ocp_values.txt"):
        v = oracle.e4m3(code)
        if math.isnan(val):
            assert math.isnan(v)
        else:
            assert v == val and math.copysign(1, v) == math.copysign(1, val), hex(code)


def test_e2m1_all_16_codes_match_spec_table():
    rows = indep.read_table("e2m1_ocp_values.txt")
    assert len(rows) == 16
    for code, val in rows:
        v = oracle.e2m1(code)
        assert v == val and math.copysign(1, v) == math.copysign(1, val), hex(code)


def test_e4m3_values_exact_in_bf16_and_f16():
    v = torch.tensor([oracle.e4m3(c) for c in range(256) if c not in (0x7F, 0xFF)],
                     dtype=torch.float64)
    assert torch.equal(v.to(torch.bfloat16).to(torch.float64), v)
    assert torch.equal(v.to(torch.float16).to(torch.float64), v)


def test_e2m1_times_e4m3_products_exact_in_f16_and_bf16():
    a = torch.tensor([oracle.e2m1(n) for n in range(16)], dtype=torch.float64)
    b = torch.tensor([oracle.e4m3(c) for c in range(256) if c not in (0x7F, 0xFF)],
                     dtype=torch.float64)
    p = (a[:, None] * b[None, :]).flatten()
    assert torch.equal(p.to(torch.float16).to(torch.float64), p)
    assert torch.equal(p.to(torch.bfloat16).to(torch.float64), p)


def test_bf16_decode_matches_torch():
    rng = np.random.default_rng(1)
    bits = rng.integers(0, 1 << 16, size=4000, dtype=np.uint16)
    bits = bits[(bits & 0x7F80) != 0x7F80]  # finite only
    ref = indep.bf16_to_f64(bits)
    got = np.array([oracle.bf16_value(int(b)) for b in bits])
    assert np.array_equal(got, ref)


def test_bf16_rounding_is_nearest_even():
    rng = np.random.default_rng(2)
    v = rng.standard_normal(5000).astype(np.float32).astype(np.float64)
    bits = oracle.to_bf16_bits(v)
    ref = torch.tensor(v, dtype=torch.float32).to(torch.bfloat16).view(torch.int16).numpy()
    assert np.array_equal(bits.view(np.int16), ref)
    # an exact tie between two bf16 neighbours goes to the even one
    lo = indep.bf16_to_f64(np.array([0x3F80], np.uint16))[0]  # 1.0
    hi = indep.bf16_to_f64(np.array([0x3F81], np.uint16))[0]
    assert oracle.to_bf16_bits(np.array([(lo + hi) / 2]))[0] == 0x3F80
    hi2 = indep.bf16_to_f64(np.array([0x3F82], np.uint16))[0]
    assert oracle.to_bf16_bits(np.array([(hi + hi2) / 2]))[0] == 0x3F82


@pytest.mark.parametrize("fmt", [1, 2])
def test_dequant_matches_independent_decoders(fmt):
    from paper_2609_11133_gb300 import synth
    from tests.util_np import weights_np
    w = weights_np(synth.make_weights(fmt, 3, 256, 128, seed=5))
    ow = oracle.ExpertWeights(w.fmt, w.E, w.H, w.I, w.w_gate, w.w_up, w.w_down, w.s_gate,
                              w.s_up, w.s_down, w.ts_gate, w.ts_up, w.ts_down)
    for which in ("gate", "up", "down"):
        for e in range(3):
            assert np.array_equal(ow.dequant(which, e), indep.dequant(w, which, e))
