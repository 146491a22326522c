"""Pins of the whole per-head schedule: Steps 1-3 with the periodic update
(Sec. 4) against the hand-worked 4x4 grid and the retention invariants."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import headkv as O
from synth import configs, gen
from _hand import load


def hand_params(c):
    return O.HeadParams(n_cond=c["n_cond"], n_image=c["n_image"], recent_w=c["recent_w"],
                        local_w=c["local_w"], period=c["period"], group_at=c["group_at"],
                        global_budget=c["global_budget"], tau=c["tau"], r_s=c["r_s"])


def test_hand_worked_grid():
    case, heads = load()
    hp = hand_params(case["config"])
    for hd in heads:
        exp = hd["expected"]
        tr = O.run_head(hp, hd["q"], hd["k"], hd["v"])
        assert tr.label == exp["label"] and tr.n_h == exp["n_h"], hd["name"]
        assert len(tr.updates) == len(exp["updates"])
        for rec, e in zip(tr.updates, exp["updates"]):
            assert rec.t_last == e["t_last"]
            assert sorted(rec.evicted.tolist()) == e["evicted"], (hd["name"], rec.t_last)
        assert tr.final_pos.tolist() == exp["final_pos"], hd["name"]


def check_invariants(hp, tr, label):
    C, w, P = hp.n_cond, hp.recent_w, hp.period
    budget = hp.global_budget if label == O.GLOBAL else w
    prev_img = None
    for rec in tr.updates:
        pos = rec.pos
        img = pos[pos >= C]
        n_img_total = rec.t_last + 1
        assert np.all(np.diff(pos) > 0)                              # order kept
        assert np.array_equal(pos[:C], np.arange(C))                 # cond kept
        newest = np.arange(C + n_img_total - min(w, n_img_total), C + n_img_total)
        assert np.isin(newest, pos).all()                            # recent kept
        if label == O.LOCAL:
            assert img.size == min(w, n_img_total)
        else:
            assert img.size == min(budget, n_img_total)
            if rec.T > hp.hist_budget:
                M = rec.T - hp.hist_budget
                assert rec.evicted.size == M
                # strata: the T history tokens before the update, oldest first
                if prev_img is None:
                    pre = np.arange(C, C + n_img_total)
                else:
                    pre = np.concatenate([prev_img, np.arange(prev_img.max() + 1, C + n_img_total)])
                hist = pre[: pre.size - min(w, pre.size)]
                assert hist.size == rec.T
                if hp.distance == O.GRID2D:
                    # the n_long farthest from the newest image token on the
                    # grid: nothing outside the subset is farther, and among
                    # equally far tokens the older are inside
                    d2 = {int(x): O.grid_d2(int(x) - C, rec.t_last, hp.row_len) for x in hist}
                    lp = set(rec.long_pos.tolist())
                    assert len(lp) == rec.n_long and lp <= set(hist.tolist())
                    for a in lp:
                        for b in set(hist.tolist()) - lp:
                            assert (d2[a], -a) > (d2[b], -b)
                    long_set = rec.long_pos
                else:
                    long_set = hist[: rec.n_long]
                    assert np.array_equal(rec.long_pos, long_set)
                in_long = np.isin(rec.evicted, long_set).sum()
                m_long = min(M // 2, rec.n_long)
                m_long = max(m_long, M - (rec.T - rec.n_long))
                assert in_long == m_long
        assert pos.size <= C + budget + P
        prev_img = img


@pytest.mark.parametrize("name", ["tiny", "janus_pro_7b", "lumina768"])
def test_retention_invariants(name):
    w = configs.ALL[name]
    w = w.with_(n_layers=1)
    hp = O.HeadParams.of(w)
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    heads = range(w.n_heads) if name == "tiny" else (0, 3, 7, 12)
    for h in heads:
        hi = gen.HeadInputs(w, 0, 0, h, pe, cq)
        tr = O.run_head(hp, hi.q, hi.k, hi.v)
        check_invariants(hp, tr, tr.label)
        # final length: C + kept history + recent + buffered tokens
        budget = hp.global_budget if tr.label == O.GLOBAL else w.recent_w
        assert tr.final_pos.size == w.n_cond + budget + tr.nbuf


def test_period_one_buffer():
    w = configs.TINY.with_(period=1, group_at=20)
    hp = O.HeadParams.of(w)
    for h in (1, 6):
        hi = gen.HeadInputs(w, 0, 0, h)
        tr = O.run_head(hp, hi.q, hi.k, hi.v)
        check_invariants(hp, tr, tr.label)
        # grouping update + one at the start of each of steps E+1 .. N-1
        assert len(tr.updates) == w.n_image - w.group_at


def test_label_injection_overrides_grouping():
    w = configs.TINY
    hp = O.HeadParams.of(w)
    hi = gen.HeadInputs(w, 0, 0, 0)                  # a local head
    tr = O.run_head(hp, hi.q, hi.k, hi.v, label=O.GLOBAL)
    assert tr.label_computed == O.LOCAL and tr.label == O.GLOBAL
    assert tr.final_pos.size == w.n_cond + hp.global_budget + tr.nbuf


@pytest.mark.parametrize("name", ["tiny", "janus_pro_7b", "lumina768"])
def test_retention_invariants_grid_distance(name):
    """The grid-distance variant (not in the paper) keeps every budget and
    always-kept class; its long-range subset is the farthest on the grid."""
    w = configs.ALL[name].with_(n_layers=1)
    hp = O.HeadParams.of(w, distance=O.GRID2D)
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    heads = range(w.n_heads) if name == "tiny" else (0, 3, 7, 12)
    for h in heads:
        hi = gen.HeadInputs(w, 0, 0, h, pe, cq)
        tr = O.run_head(hp, hi.q, hi.k, hi.v, label=O.GLOBAL if h % 2 else None)
        check_invariants(hp, tr, tr.label)
        budget = hp.global_budget if tr.label == O.GLOBAL else w.recent_w
        assert tr.final_pos.size == w.n_cond + budget + tr.nbuf


@pytest.mark.parametrize("r_s", [0.0, 1.0])
def test_grid_distance_with_one_stratum_is_raster(r_s):
    """With a single stratum the partition cannot matter: with the same
    labels the grid-distance variant retains exactly what Eq. 5 retains."""
    w = configs.ALL["janus_pro_7b"].with_(n_layers=1, r_s=r_s)
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    for h in (1, 4):
        hi = gen.HeadInputs(w, 0, 0, h, pe, cq)
        a = O.run_head(O.HeadParams.of(w), hi.q, hi.k, hi.v, label=O.GLOBAL)
        b = O.run_head(O.HeadParams.of(w, distance=O.GRID2D), hi.q, hi.k, hi.v, label=O.GLOBAL)
        assert np.array_equal(a.final_pos, b.final_pos)
        assert [u.evicted.tolist() for u in a.updates] == [u.evicted.tolist() for u in b.updates]
