"""Pins of the oracle's layer output: closed forms, brute force, invariants."""
from fractions import Fraction

import mpmath
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_11133_gb300 import synth
from tests import indep
from tests.util_np import np_, oracle_weights, weights_np

SHAPES = {1: dict(H=256, I=128), 2: dict(H=64, I=48)}


def silu(z):
    return z / (1.0 + np.exp(-z))


def ffn_dense(wn, e, xv):
    g = xv @ indep.dequant(wn, "gate", e).T
    u = xv @ indep.dequant(wn, "up", e).T
    return (silu(g) * u) @ indep.dequant(wn, "down", e).T


def inputs(fmt, E, T, seed):
    sh = SHAPES[fmt]
    w = synth.make_weights(fmt, E, sh["H"], sh["I"], seed=seed)
    x = np_(synth.make_x(T, sh["H"], seed=seed))
    wr = np_(synth.make_router(E, sh["H"], seed=seed))
    return w, x, wr


@pytest.mark.parametrize("fmt", [1, 2])
def test_one_expert_top1_is_dense_swiglu(fmt):
    w, x, wr = inputs(fmt, 1, 6, 10)
    out, ids, gates, _ = oracle.layer(oracle_weights(w), x, wr, 1)
    assert (ids == 0).all() and (gates == 1.0).all()
    ref = ffn_dense(weights_np(w), 0, indep.bf16_to_f64(x))
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())


@pytest.mark.parametrize("fmt,E,k", [(1, 6, 2), (2, 5, 3), (2, 4, 4)])
def test_sparse_layer_equals_dense_masked_formulation(fmt, E, k):
    w, x, wr = inputs(fmt, E, 5, 20 + E)
    bias = np.linspace(-0.1, 0.1, E).astype(np.float32)
    out, ids, gates, _ = oracle.layer(oracle_weights(w), x, wr, k, router_bias=bias)
    wn = weights_np(w)
    xv = indep.bf16_to_f64(x)
    logits = xv @ wr.astype(np.float64).T + bias
    ref = np.zeros_like(out)
    for t in range(x.shape[0]):
        sel = sorted(range(E), key=lambda e: (-logits[t, e], e))[:k]
        p = np.exp(logits[t, sel] - logits[t, sel].max())
        ghat = np.zeros(E)
        ghat[sel] = p / p.sum()
        for e in range(E):  # every expert, gate zero off the top-k
            ref[t] += ghat[e] * ffn_dense(wn, e, xv[t])
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12 * np.abs(ref).max())


@pytest.mark.parametrize("fmt", [1, 2])
def test_zero_code_expert_contributes_nothing(fmt):
    w, x, wr = inputs(fmt, 4, 8, 30)
    ow = oracle_weights(w)
    _, ids, gates, _ = oracle.layer(ow, x, wr, 2)
    victim = int(ids[0, 0])
    wz = weights_np(w)
    for name in ("w_gate", "w_up", "w_down"):
        getattr(wz, name)[victim] = 0
    owz = oracle_weights(wz)
    out_z = oracle.moe_tokens(owz, x, ids, gates)
    # reference: the same routing with that expert's gate set to zero
    gz = gates.copy()
    gz[ids == victim] = 0.0
    ref = oracle.moe_tokens(ow, x, ids, gz)
    np.testing.assert_array_equal(out_z, ref)


@pytest.mark.parametrize("fmt,p", [(1, 3), (1, -5), (2, 4), (2, -2)])
def test_power_of_two_down_scale_scales_output_exactly(fmt, p):
    w, x, wr = inputs(fmt, 4, 5, 40)
    ow = oracle_weights(w)
    out, ids, gates, _ = oracle.layer(ow, x, wr, 2)
    ws = weights_np(w)
    if fmt == 1:
        ws.s_down = ws.s_down * np.float32(2.0 ** p)
    else:
        ws.ts_down = ws.ts_down * np.float32(2.0 ** p)
    out2 = oracle.moe_tokens(oracle_weights(ws), x, ids, gates)
    np.testing.assert_array_equal(out2, out * 2.0 ** p)


def test_token_permutation_permutes_outputs():
    w, x, wr = inputs(1, 6, 7, 50)
    ow = oracle_weights(w)
    out, _, _, _ = oracle.layer(ow, x, wr, 2)
    perm = np.random.default_rng(0).permutation(7)
    out_p, _, _, _ = oracle.layer(ow, x[perm], wr, 2)
    np.testing.assert_array_equal(out_p, out[perm])


def test_expert_relabelling_keeps_output():
    w, x, wr = inputs(2, 5, 6, 60)
    out, _, _, _ = oracle.layer(oracle_weights(w), x, wr, 2)
    perm = np.array([3, 0, 4, 1, 2])
    wn = weights_np(w)
    for name in ("w_gate", "w_up", "w_down", "s_gate", "s_up", "s_down", "ts_gate", "ts_up",
                 "ts_down"):
        setattr(wn, name, getattr(wn, name)[perm])
    out2, _, _, _ = oracle.layer(oracle_weights(wn), x, wr[perm], 2)
    np.testing.assert_allclose(out2, out, rtol=1e-13, atol=1e-14)


def test_residual_is_added():
    w, x, wr = inputs(1, 4, 3, 70)
    ow = oracle_weights(w)
    out, ids, gates, _ = oracle.layer(ow, x, wr, 2)
    res = np_(synth.make_x(3, 256, seed=71))
    out_r = oracle.moe_tokens(ow, x, ids, gates, residual_bits=res)
    np.testing.assert_allclose(out_r, out + indep.bf16_to_f64(res), rtol=1e-15, atol=1e-15)


def test_exact_rational_reference_tiny_nvfp4():
    """H=32, I=16: every product and sum done in exact rationals, SiLU in 60 digits."""
    mpmath.mp.dps = 60
    w = synth.make_weights(2, 2, 32, 16, seed=81)
    x = np_(synth.make_x(2, 32, seed=81))
    wr = np_(synth.make_router(2, 32, seed=81))
    ow = oracle_weights(w)
    out, ids, gates, _ = oracle.layer(ow, x, wr, 1)
    wn = weights_np(w)
    xf = [[Fraction(float(v)) for v in row] for row in indep.bf16_to_f64(x)]
    for t in range(2):
        e = int(ids[t, 0])
        Wg, Wu, Wd = (indep.dequant(wn, m, e) for m in ("gate", "up", "down"))
        h = []
        for i in range(16):
            g = sum(xf[t][c] * Fraction(float(Wg[i, c])) for c in range(32))
            u = sum(xf[t][c] * Fraction(float(Wu[i, c])) for c in range(32))
            gm = mpmath.mpf(g.numerator) / g.denominator
            um = mpmath.mpf(u.numerator) / u.denominator
            h.append(gm / (1 + mpmath.e ** (-gm)) * um)
        for r in range(32):
            y = sum(h[i] * mpmath.mpf(float(Wd[r, i])) for i in range(16))
            assert abs(float(y) - out[t, r]) <= 1e-12 * max(1.0, abs(float(y)))


def test_rmsnorm_eps_and_mean_pinned_by_worked_values():
    """The pre-norm reading bf16(x / sqrt(mean(x^2) + eps)), eps = 1e-6 inside
    the root, pinned by values worked out by hand where the other readings
    differ: a constant row at 2^-10, whose mean square (2^-20) is comparable
    to eps, gives 2^-10 / sqrt(2^-20 + 1e-6) = 0.698677..., bf16 0.69921875
    (eps outside the root would give 0.99898 -> 1.0, no eps 1.0); a row with
    one element 1 and 63 zeros gives 1 / sqrt(1/64 + 1e-6) = 7.99974..., bf16
    8.0 (a sum instead of a mean would give 1.0)."""
    H = 64
    const = np.full((1, H), 2.0 ** -10)
    one = np.zeros((1, H))
    one[0, 0] = 1.0
    # both rows hold values exact in bf16: their bits are the top half of the fp32 bits
    rows = np.concatenate([const, one]).astype(np.float32)
    bits = (rows.view(np.uint32) >> 16).astype(np.uint16)
    out = indep.bf16_to_f64(oracle.rmsnorm_bf16(bits, 1e-6))
    assert (out[0] == 0.69921875).all()
    assert out[1, 0] == 8.0 and (out[1, 1:] == 0.0).all()


def test_rmsnorm_rounds_to_nearest_bf16():
    x = np_(synth.make_x(4, 64, seed=90, std=3.0))
    xn = oracle.rmsnorm_bf16(x, 1e-6)
    xv = indep.bf16_to_f64(x)
    v = xv / np.sqrt((xv ** 2).mean(axis=1, keepdims=True) + 1e-6)
    got = indep.bf16_to_f64(xn)
    # the chosen bf16 is no further from v than its two neighbours
    for d in (-1, 1):
        nb = indep.bf16_to_f64((xn.astype(np.int32) + d).astype(np.uint16))
        assert (np.abs(got - v) <= np.abs(nb - v)).all()
