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
