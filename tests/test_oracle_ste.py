"""Pins of Stratified Token Eviction (Sec. 4, Eqs. 5-6)."""
import itertools
import math

import numpy as np
import pytest

from oracle import headkv as O
from synth import configs, gen


def brute_force_evict(scores, n_long, m_long, m_near):
    """Among all eviction sets with m_long tokens from the first n_long and
    m_near from the rest, the one with the smallest total score (unique for
    distinct scores)."""
    T = len(scores)
    best, best_sum = None, None
    for ev_l in itertools.combinations(range(n_long), m_long):
        for ev_n in itertools.combinations(range(n_long, T), m_near):
            s = sum(scores[i] for i in ev_l + ev_n)
            if best_sum is None or s < best_sum:
                best, best_sum = set(ev_l + ev_n), s
    return best


@pytest.mark.parametrize("seed", range(12))
def test_matches_brute_force_enumeration(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(4, 10))
    n_long = O.ste_partition(T, 0.5)
    M = int(rng.integers(1, T))
    scores = rng.permutation(T * 3)[:T].astype(np.float32)      # distinct
    pos = np.arange(10, 10 + T)
    m_long, m_near = O.ste_quotas(M, n_long, T - n_long)
    ev = O.ste_evict(scores, pos, n_long, M)
    assert set(np.nonzero(ev)[0]) == brute_force_evict(list(scores), n_long, m_long, m_near)
    assert ev.sum() == M


def test_partition_eq5():
    assert O.ste_partition(975, 0.5) == 487
    assert O.ste_partition(6, 0.5) == 3
    assert O.ste_partition(7, 0.5) == 3
    assert O.ste_partition(10, 0.6) == 6
    assert O.ste_partition(5, 0.0) == 0 and O.ste_partition(5, 1.0) == 5


def test_quotas_half_each_and_spill():
    assert O.ste_quotas(65, 487, 488) == (32, 33)
    assert O.ste_quotas(64, 487, 488) == (32, 32)
    assert O.ste_quotas(5, 1, 10) == (1, 4)       # long too small
    assert O.ste_quotas(6, 10, 2) == (4, 2)       # near too small
    assert O.ste_quotas(0, 3, 3) == (0, 0)
    assert O.ste_quotas(7, 0, 9) == (0, 7)        # r_s = 0: one group
    assert O.ste_quotas(7, 9, 0) == (7, 0)        # r_s = 1: one group


@pytest.mark.parametrize("r_s", [0.0, 1.0])
def test_single_stratum_is_plain_lowest_m(r_s):
    rng = np.random.default_rng(7)
    for _ in range(20):
        T = int(rng.integers(5, 200))
        M = int(rng.integers(1, T))
        scores = rng.normal(size=T).astype(np.float32)
        ev = O.ste_evict(scores, np.arange(T), O.ste_partition(T, r_s), M)
        lowest = np.argpartition(scores, M - 1)[:M]
        assert set(np.nonzero(ev)[0]) == set(lowest.tolist())


def test_ties_evict_older_first():
    scores = np.zeros(8, dtype=np.float32)
    pos = np.array([3, 5, 6, 9, 11, 12, 20, 21])
    ev = O.ste_evict(scores, pos, 4, 4)            # 2 per stratum
    assert np.nonzero(ev)[0].tolist() == [0, 1, 4, 5]


def test_strata_are_independent():
    # the near group holds all the low scores; a single top-k would evict
    # only near tokens, STE still evicts M/2 from the long group
    scores = np.array([5, 6, 7, 8, 0, 1, 2, 3], dtype=np.float32)
    ev = O.ste_evict(scores, np.arange(8), 4, 4)
    assert np.nonzero(ev)[0].tolist() == [0, 1, 4, 5]


def test_fp32_scores_exact_on_integers():
    # integer inputs: every fp32 op is exact, so the decision score equals the
    # integer sum over queries and channels of q_p[d] k_j[d]
    rng = np.random.default_rng(11)
    Q = rng.integers(-8, 9, size=(5, 16)).astype(np.float32)
    K = rng.integers(-8, 9, size=(30, 16)).astype(np.float32)
    exact = np.array([sum(int(Q[p, d]) * int(K[j, d]) for p in range(5) for d in range(16))
                      for j in range(30)])
    assert np.array_equal(O.ste_scores_fp32(Q, K), exact.astype(np.float32))
    # and Eq. 6 is the same number scaled by 1/(P sqrt(d))
    np.testing.assert_allclose(O.ste_scores_eq6(Q, K), exact / (5 * 4.0), rtol=0, atol=1e-12)


def test_fp32_decision_ranks_like_eq6():
    """On model-shaped data the fp32 decision evicts the same tokens as the
    fp64 Eq. 6 scores, except where the two sides of the cut are closer than
    fp32 rounding can resolve."""
    w = configs.LUMINA_1024.with_(n_layers=1)
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    mismatches = 0
    for h in range(8):
        hi = gen.HeadInputs(w, 0, 0, h, pe, cq)
        T, P = 975, w.period
        hist = np.arange(w.n_cond, w.n_cond + T)
        Q = hi.q[1500 - P + 1: 1501]
        s32 = O.ste_scores_fp32(Q, hi.k[hist])
        s64 = O.ste_scores_eq6(Q, hi.k[hist])
        n_long = O.ste_partition(T, w.r_s)
        e32 = O.ste_evict(s32, hist, n_long, P)
        e64 = O.ste_evict(s64, hist, n_long, P)
        if not np.array_equal(e32, e64):
            mismatches += 1
            diff = np.nonzero(e32 != e64)[0]
            scale = np.abs(s64).max()
            # any disagreement must sit on a near-tie of the fp64 scores
            for i in diff:
                others = diff[diff != i]
                assert np.min(np.abs(s64[others] - s64[i])) < 1e-5 * scale
        # scaled fp32 scores track Eq. 6 closely
        np.testing.assert_allclose(s32 / (P * math.sqrt(w.head_dim)), s64,
                                   rtol=0, atol=1e-5 * np.abs(s64).max())
    assert mismatches <= 1


# Grid-distance variant of Eq. 5 (not in the paper).

def test_long_subset_2d_hand_worked():
    # row_len 4, C = 2, newest image token 9 at (2, 1); history image
    # tokens 0..5 (positions 2..7) at squared distances 5, 4, 5, 8, 2, 1.
    # The 3 farthest: token 3 (8), then tokens 0 and 2 (5; older first).
    hist = np.arange(2, 8)
    mask = O.ste_long_2d(hist, 3, 2, 4, 9)
    assert hist[mask].tolist() == [2, 4, 5]
    # raster Eq. 5 would take the oldest three: positions 2, 3, 4


def brute_force_evict_mask(scores, is_long, m_long, m_near):
    lo = [i for i in range(len(scores)) if is_long[i]]
    ne = [i for i in range(len(scores)) if not is_long[i]]
    best, best_sum = None, None
    for ev_l in itertools.combinations(lo, m_long):
        for ev_n in itertools.combinations(ne, m_near):
            s = sum(scores[i] for i in ev_l + ev_n)
            if best_sum is None or s < best_sum:
                best, best_sum = set(ev_l + ev_n), s
    return best


@pytest.mark.parametrize("seed", range(12))
def test_strata_mask_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    T = int(rng.integers(4, 10))
    is_long = rng.permutation(T) < O.ste_partition(T, 0.5)
    M = int(rng.integers(1, T))
    scores = rng.permutation(T * 3)[:T].astype(np.float32)
    pos = np.arange(10, 10 + T)
    m_long, m_near = O.ste_quotas(M, int(is_long.sum()), T - int(is_long.sum()))
    ev = O.ste_evict_strata(scores, pos, is_long, M)
    assert set(np.nonzero(ev)[0]) == brute_force_evict_mask(list(scores), is_long, m_long, m_near)


def test_strata_mask_of_the_oldest_is_eq5():
    rng = np.random.default_rng(7)
    for T in (5, 17, 64):
        scores = rng.normal(size=T).astype(np.float32)
        pos = np.sort(rng.choice(1000, size=T, replace=False))
        n_long = O.ste_partition(T, 0.5)
        for M in (1, T // 3, T - 1):
            assert np.array_equal(O.ste_evict_strata(scores, pos, np.arange(T) < n_long, M),
                                  O.ste_evict(scores, pos, n_long, M))
