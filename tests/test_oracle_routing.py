"""Pins of the oracle's router, top-k, gates and permutation."""
import numpy as np
import pytest

from oracle import oracle
from tests import indep


def brute_topk(l, k):
    return sorted(range(len(l)), key=lambda e: (-l[e], e))[:k]


@pytest.mark.parametrize("E,k", [(8, 2), (128, 8), (160, 8), (7, 7), (1, 1)])
def test_topk_matches_full_stable_sort(E, k):
    rng = np.random.default_rng(E * 31 + k)
    logits = rng.standard_normal((40, E))
    logits[::5, : E // 2] = 0.25  # crafted ties
    logits[1::7] = 1.5            # all equal rows
    ids, gates = oracle.topk(logits, k)
    for t in range(logits.shape[0]):
        ref = brute_topk(list(logits[t]), k)
        assert list(ids[t]) == ref
        sel = logits[t, ref]
        p = np.exp(sel - sel.max())
        np.testing.assert_allclose(gates[t], p / p.sum(), rtol=1e-14, atol=0)
        assert abs(gates[t].sum() - 1.0) < 1e-14


def test_all_equal_logits_give_first_k_and_uniform_gates():
    ids, gates = oracle.topk(np.zeros((3, 16)), 4)
    assert (ids == np.arange(4)).all()
    assert np.allclose(gates, 0.25, rtol=0, atol=1e-15)


def test_negative_zero_ties_with_positive_zero():
    l = np.array([[-1.0, -0.0, 0.0, -2.0]])
    ids, _ = oracle.topk(l, 2)
    assert list(ids[0]) == [1, 2]


def test_no_renorm_gives_full_softmax_probabilities():
    rng = np.random.default_rng(3)
    l = rng.standard_normal((5, 12))
    ids, gates = oracle.topk(l, 3, renorm=False)
    for t in range(5):
        p = np.exp(l[t] - l[t].max())
        p /= p.sum()
        np.testing.assert_allclose(gates[t], p[ids[t]], rtol=1e-14)


def test_single_expert_gate_is_one():
    ids, gates = oracle.topk(np.array([[0.3], [-4.0]]), 1)
    assert (ids == 0).all() and (gates == 1.0).all()


def test_router_logits_match_float64_matmul():
    rng = np.random.default_rng(4)
    T, H, E = 5, 96, 7
    xb = (rng.standard_normal((T, H)).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    wr = (rng.standard_normal((E, H)) * 0.02).astype(np.float32)
    bias = rng.standard_normal(E).astype(np.float32)
    got = oracle.router_logits(xb, wr, bias)
    ref = indep.bf16_to_f64(xb) @ wr.astype(np.float64).T + bias
    np.testing.assert_allclose(got, ref, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("T,k,E", [(1, 8, 128), (37, 8, 160), (4, 2, 8), (64, 1, 1), (5, 3, 3)])
def test_permute_matches_stable_argsort(T, k, E):
    rng = np.random.default_rng(T + k + E)
    ids = np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)
    counts, offsets, srt, inv, active = oracle.permute(ids, E)
    flat = ids.reshape(-1)
    assert np.array_equal(counts, np.bincount(flat, minlength=E))
    assert np.array_equal(offsets, np.concatenate([[0], np.cumsum(counts)]))
    assert np.array_equal(srt, np.argsort(flat, kind="stable"))
    assert np.array_equal(inv[srt], np.arange(T * k))
    act = np.nonzero(counts)[0]
    assert active[0] == act.size and np.array_equal(active[1:1 + act.size], act)
