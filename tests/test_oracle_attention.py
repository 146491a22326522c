"""Pins of the oracle's Eq. 1 (single-query softmax attention) to closed
forms and to the uncompressed causal attention it must reproduce."""
import math
from fractions import Fraction

import numpy as np
import pytest

from oracle import headkv as O
from synth import configs, gen


def test_equal_keys_give_mean_of_values():
    rng = np.random.default_rng(1)
    K = np.tile(rng.normal(size=(1, 16)), (9, 1))
    V = rng.normal(size=(9, 16))
    q = rng.normal(size=16)
    np.testing.assert_allclose(O.attention(q, K, V), V.mean(axis=0), rtol=0, atol=1e-14)


def test_dominant_key_selects_its_value():
    D = 64
    rng = np.random.default_rng(2)
    K = np.zeros((12, D))
    K[7, 0] = 50.0 * math.sqrt(D)          # logit 50 above the rest
    q = np.zeros(D)
    q[0] = 1.0
    V = rng.normal(size=(12, D))
    np.testing.assert_allclose(O.attention(q, K, V), V[7], rtol=0, atol=1e-19 * 12 + 1e-15)


def test_two_tokens_is_logistic_mix():
    # softmax over two logits a, b weights the first value by 1/(1+e^(b-a))
    D = 4
    q = np.array([1.0, 0.0, 0.0, 0.0])
    K = np.array([[3.0, 0, 0, 0], [1.0, 0, 0, 0]])   # logits 1.5 and 0.5
    V = np.array([[1.0, 0, 0, 0], [0.0, 1, 0, 0]])
    wgt = 1.0 / (1.0 + math.exp(-1.0))
    np.testing.assert_allclose(O.attention(q, K, V), [wgt, 1 - wgt, 0, 0], rtol=0, atol=1e-15)


def test_scaling_is_one_over_sqrt_d():
    # same logits reached through different d: q.k = 2 sqrt(d) -> logit 2
    for D in (1, 4, 64, 128):
        q = np.zeros(D); q[0] = 2.0 * math.sqrt(D)
        K = np.zeros((2, D)); K[0, 0] = 1.0
        V = np.array([[1.0] + [0.0] * (D - 1), [0.0] * D])
        w = 1.0 / (1.0 + math.exp(-2.0))
        assert abs(O.attention(q, K, V)[0] - w) < 1e-15


def test_permutation_invariance():
    rng = np.random.default_rng(3)
    K = rng.normal(size=(30, 8)); V = rng.normal(size=(30, 8)); q = rng.normal(size=8)
    perm = rng.permutation(30)
    np.testing.assert_allclose(O.attention(q, K, V), O.attention(q, K[perm], V[perm]), atol=1e-14)


def test_empty_cache_gives_zero():
    assert np.all(O.attention(np.ones(4), np.zeros((0, 4)), np.zeros((0, 4))) == 0)


@pytest.mark.parametrize("label", [O.GLOBAL])
def test_full_budget_reproduces_dense_causal_attention(label):
    """rho = 1: a global head keeps all N image tokens, nothing is ever
    evicted, and every step's output equals the uncompressed causal attention
    (computed here as one masked matrix product)."""
    w = configs.TINY.with_(rho=Fraction(1, 1))
    hp = O.HeadParams.of(w)
    assert hp.global_budget == w.n_image
    for h in (0, 5):
        hi = gen.HeadInputs(w, 0, 0, h)
        tr = O.run_head(hp, hi.q, hi.k, hi.v, label=label, record=range(w.n_image))
        dense = O.dense_causal_attention(hi.q, hi.k, hi.v, w.n_cond)
        got = np.stack([tr.outputs[t] for t in range(w.n_image)])
        np.testing.assert_allclose(got, dense, rtol=0, atol=1e-12)
        assert all(u.evicted.size == 0 for u in tr.updates)
        assert tr.final_pos.size == w.n_cond + w.n_image
