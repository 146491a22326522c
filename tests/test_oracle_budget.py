"""Pins of the budget allocation (Sec. 5.1) and the arena layout."""
from fractions import Fraction

import numpy as np

from oracle import headkv as O


def test_global_budget_matches_table3_B_column():
    # Table 3 prints B for each model and rho: 576/4 = 144, 576/6 = 96,
    # 576/8 = 72 (LlamaGen-XL, Janus-Pro-7B, N = 576) and 294 (Lumina-mGPT-768,
    # N = 2352, rho = 1/8); rho = 1 keeps all N.
    assert O.global_budget(Fraction(1, 4), 576) == 144
    assert O.global_budget(Fraction(1, 6), 576) == 96
    assert O.global_budget(Fraction(1, 8), 576) == 72
    assert O.global_budget(Fraction(1, 8), 2352) == 294
    assert O.global_budget(Fraction(1, 1), 2352) == 2352
    assert O.global_budget(Fraction(1, 6), 4160) == 693    # floor(693.33)


def test_local_budget_is_smaller():
    assert O.head_budget(O.LOCAL, 144, 48) == 48 < O.head_budget(O.GLOBAL, 144, 48)


def test_arena_layout_hand_example():
    # labels L G G L with C = 3, B_g = 10, w = 4, P = 2:
    # caps 3+4+2 = 9, 3+10+2 = 15, 15, 9; offsets 0, 9, 24, 39; total 48
    budget, cap, off, total = O.arena_layout([0, 1, 1, 0], 3, 10, 4, 2)
    assert list(budget) == [4, 10, 10, 4]
    assert list(cap) == [9, 15, 15, 9]
    assert list(off) == [0, 9, 24, 39]
    assert total == 48


def test_arena_layout_closed_form_total():
    rng = np.random.default_rng(0)
    labels = rng.integers(0, 2, size=1000)
    C, B_g, w, P = 128, 1040, 130, 65
    _, cap, off, total = O.arena_layout(labels, C, B_g, w, P)
    g = int(labels.sum())
    assert total == g * (C + B_g + P) + (1000 - g) * (C + w + P)
    assert np.all(off[1:] == off[:-1] + cap[:-1]) and off[0] == 0


def test_redistributed_budgets_hand_example():
    # one group L G G L G, B_g = 10, w = 4: the two local heads leave
    # 2 * (10 - 4) = 12 tokens; three global heads get 4 each; total 5 * 10
    b = O.redistributed_budgets([0, 1, 1, 0, 1], 10, 4)
    assert list(b) == [4, 14, 14, 4, 14] and b.sum() == 50
    b = O.redistributed_budgets([0, 1, 0, 1], 10, 4)     # 12 left: 6 each
    assert list(b) == [4, 16, 4, 16]
    b = O.redistributed_budgets([1, 0, 1], 11, 4)     # 7 left: 4 and 3
    assert list(b) == [15, 4, 14] and b.sum() == 33


def test_redistributed_budgets_invariants():
    rng = np.random.default_rng(3)
    for _ in range(200):
        H = int(rng.integers(1, 40))
        lab = rng.integers(0, 2, size=H)
        B_g = int(rng.integers(5, 200))
        w = int(rng.integers(1, B_g + 1))
        b = O.redistributed_budgets(lab, B_g, w)
        assert (b[lab == 0] == w).all()                    # local heads keep w
        g = b[lab == 1]
        if g.size:
            assert b.sum() == H * B_g                      # the group's total as uniform B_g
            assert g.min() >= B_g and g.max() - g.min() <= 1
            # the remainder goes to the global heads of lowest index
            assert (np.diff(g) <= 0).all()
        else:
            assert b.sum() == H * w


def test_arena_layout_grouped_matches_paper_without_locals():
    # every head global: the redistribution changes nothing
    lab = np.ones(64, dtype=np.int64)
    a = O.arena_layout(lab, 8, 30, 6, 4)
    b = O.arena_layout(lab, 8, 30, 6, 4, group=16)
    assert all(np.array_equal(x, y) for x, y in zip(a[:3], b[:3])) and a[3] == b[3]
    # groups are independent
    lab = np.array([0, 1, 1, 1, 0, 0, 0, 1])
    b, cap, off, total = O.arena_layout(lab, 2, 10, 4, 3, group=4)
    assert list(b) == [4, 12, 12, 12, 4, 4, 4, 28]
    assert total == int((2 + b + 3).sum())
