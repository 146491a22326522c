"""Pins of the head-grouping rule (Sec. 4, Step 2)."""
import math

import numpy as np
import pytest

from oracle import headkv as O
from synth import configs, gen


def test_uniform_attention_count_is_ceil_tau_len():
    # q = 0 makes every logit equal: the newest n tokens carry n/len
    for n, tau in ((47, 0.9), (100, 0.85), (13, 0.95), (64, 0.9)):
        K = np.random.default_rng(n).normal(size=(n, 8))
        n_h, cum = O.grouping_count(np.zeros(8), K, tau)
        expect = math.ceil(tau * n)
        if abs(tau * n - round(tau * n)) < 1e-9:   # exact multiple: fp boundary
            assert n_h in (expect, expect + 1)
        else:
            assert n_h == expect


def test_dominant_newest_token_is_local():
    D = 64
    K = np.zeros((40, D)); K[-1, 0] = 30 * math.sqrt(D)
    q = np.zeros(D); q[0] = 1.0
    n_h, _ = O.grouping_count(q, K, 0.9)
    assert n_h == 1 and O.classify(n_h, 32) == O.LOCAL


def test_hand_worked_masses():
    # D = 1, logits ln(p) give attention exactly proportional to p
    p = np.array([0.04, 0.06, 0.1, 0.3, 0.5])          # oldest .. newest
    K = np.log(p)[:, None]
    q = np.array([1.0])
    # backward masses 0.5, 0.8, 0.9, 0.96, 1.0
    assert O.grouping_count(q, K, 0.85)[0] == 3
    assert O.grouping_count(q, K, 0.75)[0] == 2
    assert O.grouping_count(q, K, 0.95)[0] == 4
    assert O.grouping_count(q, K, 0.45)[0] == 1
    # w_loc = 3: n_h = 3 is not below it -> global; w_loc = 4 -> local
    assert O.classify(3, 3) == O.GLOBAL and O.classify(3, 4) == O.LOCAL
    _, cum = O.grouping_count(q, K, 0.85)
    assert abs(O.label_margin(cum, 0.85, 4) - 0.05) < 1e-12   # mass of newest 3 = 0.9


def test_backward_accumulation_starts_at_newest():
    # a heavy OLD token must not make the head local
    D = 64
    K = np.zeros((50, D)); K[0, 0] = 30 * math.sqrt(D)
    q = np.zeros(D); q[0] = 1.0
    n_h, _ = O.grouping_count(q, K, 0.9)
    assert n_h == 50 and O.classify(n_h, 32) == O.GLOBAL


def test_hand_case_labels():
    from _hand import load
    case, heads = load()
    c = case["config"]
    for hd in heads:
        t = c["group_at"] - 1
        K = hd["k"][: c["n_cond"] + t + 1]
        n_h, cum = O.grouping_count(hd["q"][t], K, c["tau"])
        assert n_h == hd["expected"]["n_h"]
        assert O.classify(n_h, c["local_w"]) == hd["expected"]["label"]


def test_tiny_generator_gives_intended_head_types():
    """Tiny workload: beta = 4 heads (0-3) local, beta = 0.3 heads (4-7) global."""
    w = configs.TINY
    hp = O.HeadParams.of(w)
    labels = []
    for h in range(w.n_heads):
        hi = gen.HeadInputs(w, 0, 0, h)
        tr = O.run_head(hp, hi.q, hi.k, hi.v, stop_after=w.group_at - 1)
        labels.append(tr.label_computed)
        assert tr.margin > 1e-3
    assert labels == [0, 0, 0, 0, 1, 1, 1, 1]


# Multi-query variant (not in the paper): P buffered queries, each over the
# cache as it stood at its own step, attention averaged.

def test_multi_query_with_one_query_is_step_2():
    rng = np.random.default_rng(11)
    for n in (5, 40, 300):
        K = rng.normal(size=(n, 16))
        q = rng.normal(size=16) * 3
        a = O.grouping_count(q, K, 0.9)
        b = O.grouping_count_multi(q[None, :], K, 0.9)
        assert a[0] == b[0] and np.array_equal(a[1], b[1])


def test_multi_query_uniform_closed_form():
    # zero queries: query p spreads 1/m_p over its m_p = n - (P-1-p) keys, so
    # key j (0-based) gets (1/P) * sum over the queries that see it of 1/m_p
    n, P, tau = 20, 4, 0.9
    K = np.random.default_rng(2).normal(size=(n, 8))
    _, cum = O.grouping_count_multi(np.zeros((P, 8)), K, tau)
    pbar = np.zeros(n)
    for p in range(P):
        m = n - (P - 1 - p)
        pbar[:m] += 1.0 / m
    pbar /= P
    assert np.allclose(cum, np.cumsum(pbar[::-1]), rtol=0, atol=1e-15)
    assert abs(cum[-1] - 1.0) < 1e-15
    # the newest key is seen by the current query only: mass 1/(P n)
    assert abs(cum[0] - 1.0 / (P * n)) < 1e-15


def test_multi_query_older_queries_do_not_see_newer_keys():
    # the current query attends only to the newest key; an older query sees
    # every key but the newest and puts its mass on the oldest: the average
    # is half on each end
    D, n = 8, 10
    K = np.zeros((n, D))
    K[-1, 0] = 40 * math.sqrt(D)
    K[0, 1] = 40 * math.sqrt(D)
    Q = np.zeros((2, D)); Q[1, 0] = 1.0; Q[0, 1] = 1.0
    n_h, cum = O.grouping_count_multi(Q, K, 0.9)
    assert abs(cum[0] - 0.5) < 1e-12 and abs(cum[-2] - 0.5) < 1e-12
    assert n_h == n            # tau needs the oldest key too: global for any w_loc <= n


# Grid-distance variant (not in the paper): the count runs outward from the
# current token by squared distance on the image grid.

def test_grid_distance_hand_values():
    assert O.grid_d2(6, 6, 4) == 0
    assert O.grid_d2(6, 5, 4) == 1 and O.grid_d2(6, 2, 4) == 1     # left, above
    assert O.grid_d2(6, 0, 4) == 5                                 # one up, two left
    assert O.grid_d2(0, 15, 4) == 18                               # opposite corners of 4x4


def test_count_order_2d_hand_worked():
    # row_len 4, two conditioning tokens, image tokens 0..6; the newest (6)
    # sits at (1, 2). Squared distances: 5 and 2 -> 1 (newer first: 5, 2),
    # 3 and 1 -> 2 (3, 1), 4 -> 4, 0 -> 5; then conditioning 1, 0.
    # Image token i has position i + 2.
    order = O.count_order_2d(9, 2, 4)
    assert order.tolist() == [8, 7, 4, 5, 3, 6, 2, 1, 0]


def test_grid_count_sees_the_token_above_as_adjacent():
    # row_len 5, one conditioning token, image tokens 0..7: the newest (7)
    # at (1, 2); all attention on image token 2, directly above it. Raster:
    # the count reaches it after 6 tokens (7, 6, 5, 4, 3, 2): global for
    # w_loc = 4. Grid: 7, then the distance-1 tokens 6 (left) and 2 (above):
    # 3 tokens, local.
    D, C, row, n = 8, 1, 5, 9
    K = np.zeros((n, D))
    K[C + 2, 0] = 60 * math.sqrt(D)
    q = np.zeros(D); q[0] = 1.0
    n_r, _ = O.grouping_count(q, K, 0.9)
    n_g, _ = O.grouping_count_2d(q, K, 0.9, C, row)
    assert n_r == 6 and n_g == 3
    assert O.classify(n_r, 4) == O.GLOBAL and O.classify(n_g, 4) == O.LOCAL


def test_grid_count_uniform_equals_raster():
    rng = np.random.default_rng(4)
    for n, C, row in ((31, 3, 7), (101, 1, 24)):   # tau * n not an integer
        K = rng.normal(size=(n, 16))
        a = O.grouping_count(np.zeros(16), K, 0.9)
        b = O.grouping_count_2d(np.zeros(16), K, 0.9, C, row)
        assert a[0] == b[0] == math.ceil(0.9 * n - 1e-12)
        assert np.allclose(a[1], b[1], rtol=0, atol=1e-13)


def test_grid_count_multi_with_one_query():
    rng = np.random.default_rng(5)
    K = rng.normal(size=(40, 16))
    q = rng.normal(size=16) * 3
    a = O.grouping_count_2d(q, K, 0.9, 4, 6)
    b = O.grouping_count_multi_2d(q[None, :], K, 0.9, 4, 6)
    assert a[0] == b[0] and np.array_equal(a[1], b[1])


def test_count_margin_hand_worked():
    """The n_h decision's distance from tau: the two cumulative masses around
    the cut (hand-worked)."""
    cum = np.array([0.5, 0.85, 0.95, 1.0])
    assert O.count_margin(cum, 0.9, 3) == pytest.approx(0.05)   # 0.95 - 0.9 vs 0.9 - 0.85
    assert O.count_margin(cum, 0.88, 3) == pytest.approx(0.03)  # 0.88 - 0.85
    assert O.count_margin(cum, 0.4, 1) == pytest.approx(0.1)    # cum[0] - tau; no token below
    assert O.count_margin(cum, 0.02, 1) == pytest.approx(0.02)  # the empty prefix: tau - 0
    # consistent with grouping_count on real weights: the cut sits where cum crosses tau
    rng = np.random.default_rng(3)
    for _ in range(20):
        q, K = rng.normal(size=4), rng.normal(size=(30, 4)) * 3
        n_h, cum = O.grouping_count(q, K, 0.9)
        m = O.count_margin(cum, 0.9, n_h)
        assert cum[n_h - 1] >= 0.9 and (n_h == 1 or cum[n_h - 2] < 0.9)
        assert m == pytest.approx(min(cum[n_h - 1] - 0.9, 0.9 - (cum[n_h - 2] if n_h > 1 else 0)))
