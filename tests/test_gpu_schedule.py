"""The whole decode path through the C-ABI against the oracle: identification,
budgets, STE with in-place compaction, and decode attention, step by step.

* the hand-worked 4x4 grid (labels, n_h, positions after every update);
* Tiny, every step and every head (outputs within 1e-5, positions exact);
* each model shape cut to 2 layers x 2 sequences, every head (positions
  exact at every update, outputs within 2e-3 at sampled steps)."""
import numpy as np
import pytest

from oracle import headkv as O
from synth import configs, gen

from _gpu_util import (LABEL_TIE, check_labels, flat, oracle_heads, oracle_labels, run_gpu)
from _hand import load as load_hand

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-5, "bf16": 2e-3}


class HandProvider:
    def __init__(self, heads, C, device):
        import torch
        self.torch = torch
        self.q = torch.from_numpy(np.stack([h["q"] for h in heads], 1)).to(device)   # [N][H][D]
        self.k = torch.from_numpy(np.stack([h["k"] for h in heads], 0)).to(device)   # [H][C+N][D]
        self.v = torch.from_numpy(np.stack([h["v"] for h in heads], 0)).to(device)
        self.C = C

    def cond(self, kc, vc, layer, stream=0):
        kc[0].copy_(self.k[:, : self.C])
        vc[0].copy_(self.v[:, : self.C])

    def image(self, q, k, v, l0, nl, t0, nt, stream=0):
        for tt in range(nt):
            t = t0 + tt
            q[tt, 0, 0].copy_(self.q[t]) if q.dim() == 5 else q[0, 0].copy_(self.q[t])
            k[0, 0].copy_(self.k[:, self.C + t])
            v[0, 0].copy_(self.v[:, self.C + t])


@pytest.mark.parametrize("fused", [True, False])
def test_hand_worked_grid_on_gpu(fused):
    import torch
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    from paper_2605_20600_gb300.runner import generate
    case, heads = load_hand()
    c = case["config"]
    cfg = H.make_config(n_layers=1, n_seqs=1, n_heads=2, head_dim=c["head_dim"], dtype="fp32",
                        n_cond=c["n_cond"], n_image=c["n_image"], row_len=c["row_len"],
                        recent_w=c["recent_w"], local_w=c["local_w"], period=c["period"],
                        group_at=c["group_at"], global_budget=c["global_budget"], tau=c["tau"],
                        r_s=c["r_s"])
    eng = Engine(cfg, "cuda")
    pos_at, outs = {}, {}

    def on_step(t, out):
        cc = eng.cache
        off, ln = cc.off.cpu().numpy(), cc.len.cpu().numpy()
        pos_at[t] = [np.sort(cc.pos[int(off[h]): int(off[h]) + int(ln[h])].cpu().numpy())
                     for h in range(2)]
        outs[t] = out.cpu().numpy()[0, 0]

    generate(eng, HandProvider(heads, c["n_cond"], "cuda"), on_step=on_step, fused=fused,
             identify="separate")
    eng.check()
    labels, nh = eng.labels.cpu().numpy(), eng.n_h.cpu().numpy()
    hp = O.HeadParams(n_cond=c["n_cond"], n_image=c["n_image"], recent_w=c["recent_w"],
                      local_w=c["local_w"], period=c["period"], group_at=c["group_at"],
                      global_budget=c["global_budget"], tau=c["tau"], r_s=c["r_s"])
    for h, hd in enumerate(heads):
        exp = hd["expected"]
        assert int(labels[h]) == exp["label"] and int(nh[h]) == exp["n_h"], hd["name"]
        # after the update that ran at the start of step t_last+1 the cache
        # holds the survivors plus the new token t_last+1
        for u in exp["updates"][1:]:
            t = u["t_last"] + 1
            assert not set(u["evicted"]) & set(pos_at[t][h].tolist()), (hd["name"], t)
        final = np.concatenate([pos_at[c["n_image"] - 1][h]])
        assert final.tolist() == exp["final_pos"], hd["name"]
        tr = O.run_head(hp, hd["q"], hd["k"], hd["v"], record=range(c["n_image"]),
                        record_pos=range(c["n_image"]))
        for t in range(c["n_image"]):
            assert np.array_equal(pos_at[t][h], tr.pos_at[t]), (hd["name"], t)
            assert np.abs(outs[t][h] - tr.outputs[t]).max() < 1e-5, (hd["name"], t)


def test_hand_worked_grid_fused_identification():
    """The grouping step's decode with the head types decided in the same
    pass gives the hand-worked labels (4x4 grid, D = 2, integer keys)."""
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    from paper_2605_20600_gb300.runner import generate
    case, heads = load_hand()
    c = case["config"]
    cfg = H.make_config(n_layers=1, n_seqs=1, n_heads=2, head_dim=c["head_dim"], dtype="fp32",
                        n_cond=c["n_cond"], n_image=c["n_image"], row_len=c["row_len"],
                        recent_w=c["recent_w"], local_w=c["local_w"], period=c["period"],
                        group_at=c["group_at"], global_budget=c["global_budget"], tau=c["tau"],
                        r_s=c["r_s"])
    eng = Engine(cfg, "cuda")
    generate(eng, HandProvider(heads, c["n_cond"], "cuda"), last_step=c["group_at"] - 1,
             fused=True, identify="fused")
    eng.check()
    labels = eng.labels.cpu().numpy()
    for h, hd in enumerate(heads):
        assert int(labels[h]) == hd["expected"]["label"], hd["name"]


@pytest.mark.parametrize("fused,identify,distance", [
    (True, "separate", O.RASTER), (False, "separate", O.RASTER), (True, "fused", O.RASTER),
    (True, "multi", O.RASTER),
    # the grid-distance variants of Step 2 and Eq. 5
    (True, "separate", O.GRID2D), (False, "separate", O.GRID2D)])
def test_tiny_every_step_every_head(fused, identify, distance):
    w = configs.TINY
    N = w.n_image
    heads = [(0, 0, h) for h in range(w.n_heads)]
    outs, poss, labels, nh, eng = run_gpu(w, out_steps=range(N), pos_steps=range(N),
                                          pos_heads=[flat(w, *x) for x in heads], fused=fused,
                                          identify=identify, distance_mode=distance)
    lab = oracle_labels(w, [0], [0], multi=identify == "multi", distance=distance)
    ties = check_labels(w, labels, nh, lab, "tiny")
    assert not ties
    assert labels.tolist() == [0, 0, 0, 0, 1, 1, 1, 1]
    tr = oracle_heads(w, heads, labels, record=range(N), record_pos=range(N), distance=distance)
    worst = 0.0
    for (s, l, h) in heads:
        t_r = tr[(s, l, h)]
        i = flat(w, s, l, h)
        for t in range(N):
            assert np.array_equal(poss[t][i], t_r.pos_at[t]), (h, t)
            worst = max(worst, float(np.abs(outs[t][l, s, h] - t_r.outputs[t]).max()))
    assert worst <= TOL["fp32"], worst


def sampled_steps(w, rng, extra=12):
    E, P, N = w.group_at, w.period, w.n_image
    s = {0, E - 2, E - 1, E, E + 1, N - 1}
    s |= {t for t in range(E, N, P)} | {t for t in range(E + P - 1, N, P)}
    s |= set(rng.integers(0, N, size=extra).tolist())
    return sorted(x for x in s if 0 <= x < N)


REDUCED = [("lumina768", "1/4", True, "separate"), ("lumina1024", "1/4", True, "separate"),
           ("lumina1024", "1/6", True, "separate"), ("lumina1024", "1/8", True, "separate"),
           ("llamagen_xl", "1/6", True, "separate"), ("janus_pro_7b", "1/8", True, "separate"),
           ("lumina1024", "1/8", False, "separate"), ("llamagen_xl", "1/6", False, "separate"),
           # the head types decided inside the grouping token's decode step
           ("lumina1024", "1/4", True, "fused"), ("llamagen_xl", "1/6", True, "fused"),
           ("janus_pro_7b", "1/8", True, "fused"),
           # the head types from the recent queries' averaged attention
           ("lumina768", "1/4", True, "multi"), ("janus_pro_7b", "1/8", True, "multi")]


@pytest.mark.parametrize("name,rho,fused,identify", REDUCED)
def test_model_shapes_two_layers_two_seqs(name, rho, fused, identify):
    from fractions import Fraction
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2, rho=Fraction(rho))
    rng = np.random.default_rng(42)
    steps = sampled_steps(w, rng)
    heads = [(s, l, h) for l in range(w.n_layers) for s in range(w.n_seqs) for h in range(w.n_heads)]
    outs, poss, labels, nh, eng = run_gpu(w, out_steps=steps, pos_steps=steps,
                                          pos_heads=[flat(w, *x) for x in heads], fused=fused,
                                          identify=identify)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs), multi=identify == "multi")
    ties = check_labels(w, labels, nh, lab, name)
    assert len(ties) <= 2, ties
    g = float((labels == 1).mean())
    assert 0.2 < g < 0.8, g                       # both head types present
    tr = oracle_heads(w, heads, labels, record=steps, record_pos=steps)
    worst = 0.0
    for (s, l, h) in heads:
        t_r, i = tr[(s, l, h)], flat(w, s, l, h)
        for t in steps:
            assert np.array_equal(poss[t][i], t_r.pos_at[t]), (name, s, l, h, t)
            worst = max(worst, float(np.abs(outs[t][l, s, h] - t_r.outputs[t]).max()))
        # retained budget after the last update
        budget = O.global_budget(w.rho, w.n_image) if labels[i] == 1 else w.recent_w
        assert poss[w.n_image - 1][i].size == w.n_cond + budget + t_r.nbuf
    assert worst <= TOL[w.dtype], worst


@pytest.mark.parametrize("name,rho", [("lumina768", "1/4"), ("llamagen_xl", "1/6"),
                                      ("janus_pro_7b", "1/8")])
def test_grid_distance_two_layers_two_seqs(name, rho):
    """The grid-distance variants (not in the paper): head types counted
    outward on the image grid and Eq. 5's long-range subset the farthest on
    it; labels, n_h, positions and outputs against the oracle run the same
    way."""
    from fractions import Fraction
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2, rho=Fraction(rho))
    steps = sampled_steps(w, np.random.default_rng(43))
    heads = [(s, l, h) for l in range(w.n_layers) for s in range(w.n_seqs) for h in range(w.n_heads)]
    outs, poss, labels, nh, eng = run_gpu(w, out_steps=steps, pos_steps=steps,
                                          pos_heads=[flat(w, *x) for x in heads],
                                          distance_mode=O.GRID2D)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs), distance=O.GRID2D)
    ties = check_labels(w, labels, nh, lab, f"{name} grid")
    assert len(ties) <= 2, ties
    tr = oracle_heads(w, heads, labels, record=steps, record_pos=steps, distance=O.GRID2D)
    worst = 0.0
    for (s, l, h) in heads:
        t_r, i = tr[(s, l, h)], flat(w, s, l, h)
        for t in steps:
            assert np.array_equal(poss[t][i], t_r.pos_at[t]), (name, s, l, h, t)
            worst = max(worst, float(np.abs(outs[t][l, s, h] - t_r.outputs[t]).max()))
    assert worst <= TOL[w.dtype], worst


def test_export_state_matches_the_cache():
    """hkv_export_state returns the layer's counters, labels and live
    positions (segment order) as the cache arrays hold them, through the
    dense phase, grouping and compressed decode."""
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth
    from _gpu_util import cfg_of
    w = configs.TINY
    eng = Engine(cfg_of(H, w), "cuda")
    n = w.n_seqs * w.n_heads
    seen = []

    def on_step(t, out):
        if t % 29 != 3 and t != w.group_at - 1 and t != w.n_image - 1:
            return
        cc = eng.cache
        for layer in range(w.n_layers):
            st = H.hkv_export_state(eng.cfg, cc.c, layer)
            sl = slice(layer * n, (layer + 1) * n)
            for k in ("label", "len", "nbuf", "ntok"):
                assert np.array_equal(st[k], getattr(cc, k)[sl].cpu().numpy()), (t, k)
            off, ln = cc.off[sl].cpu().numpy(), cc.len[sl].cpu().numpy()
            pos = cc.pos.cpu().numpy()
            for h in range(n):
                assert np.array_equal(st["pos"][h], pos[off[h]: off[h] + ln[h]]), (t, h)
        seen.append(t)

    generate(eng, DeviceSynth(w, "cuda"), on_step=on_step)
    eng.check()
    assert len(seen) >= 8 and w.group_at - 1 in seen


def test_export_state_capacity():
    import ctypes
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    from _gpu_util import cfg_of
    w = configs.TINY
    eng = Engine(cfg_of(H, w), "cuda")
    cc = eng.cache
    cc.len.fill_(3)
    cc.off.copy_(cc.off.new_tensor(list(range(0, 8 * 40, 40))))
    out = np.zeros(23, np.int32)
    cnt = ctypes.c_int64(0)
    f = H.lib().hkv_export_state
    args = (ctypes.byref(eng.cfg), ctypes.byref(cc.c), 0, None, None, None, None)
    assert f(*args, out.ctypes.data, 23, ctypes.byref(cnt), None) == H.HKV_ERR_CAPACITY
    assert cnt.value == 24
    big = np.zeros(24, np.int32)
    assert f(*args, big.ctypes.data, 24, ctypes.byref(cnt), None) == 0
    assert np.array_equal(big, cc.pos.cpu().numpy()[np.add.outer(np.arange(0, 320, 40), np.arange(3)).ravel()])
    cc.len[2] = -1
    assert f(*args, None, 0, ctypes.byref(cnt), None) == H.HKV_ERR_BOUNDS


@pytest.mark.parametrize("mode", [0, 1])
def test_budgets_match_the_oracle(mode):
    """hkv_allocate_budgets against the oracle's arena layout, both budget
    rules (cfg.budget_mode), on the Lumina-1024 head count with random labels (one group all
    local, one all global)."""
    import torch
    from paper_2605_20600_gb300 import hkv as H
    from _gpu_util import cfg_of
    w = configs.LUMINA_1024
    cfg = cfg_of(H, w, mode)
    n = w.n_layers * w.n_seqs * w.n_heads
    rng = np.random.default_rng(5 + mode)
    lab = rng.integers(0, 2, n).astype(np.uint8)
    lab[: w.n_heads] = 0
    lab[w.n_heads: 2 * w.n_heads] = 1
    dev = torch.device("cuda")
    lab_t = torch.from_numpy(lab).to(dev)
    budget = torch.empty(n, dtype=torch.int32, device=dev)
    cap = torch.empty(n, dtype=torch.int32, device=dev)
    off = torch.empty(n, dtype=torch.int64, device=dev)
    total = H.hkv_allocate_budgets(cfg, lab_t, budget, cap, off)
    B_g = O.global_budget(w.rho, w.n_image)
    ob, ocap, ooff, ototal = O.arena_layout(lab, w.n_cond, B_g, w.recent_w, w.period,
                                            group=w.n_heads if mode else 0)
    assert np.array_equal(budget.cpu().numpy(), ob)
    assert np.array_equal(cap.cpu().numpy(), ocap)
    assert np.array_equal(off.cpu().numpy(), ooff)
    assert total == ototal


@pytest.mark.parametrize("name,rho", [("lumina1024", "1/8"), ("llamagen_xl", "1/6")])
def test_model_shapes_redistributed_budgets(name, rho):
    """The aggregate-preserving budgets through the whole path: every global
    head runs STE with its own history budget; positions exact against the
    oracle with the same per-head budgets, outputs within tolerance."""
    from fractions import Fraction
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2, rho=Fraction(rho))
    rng = np.random.default_rng(43)
    steps = sampled_steps(w, rng)
    heads = [(s, l, h) for l in range(w.n_layers) for s in range(w.n_seqs) for h in range(w.n_heads)]
    outs, poss, labels, nh, eng = run_gpu(w, out_steps=steps, pos_steps=steps,
                                          pos_heads=[flat(w, *x) for x in heads], budget_mode=1)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs))
    check_labels(w, labels, nh, lab, name)
    B_g = O.global_budget(w.rho, w.n_image)
    budgets = O.arena_layout(labels, w.n_cond, B_g, w.recent_w, w.period, group=w.n_heads)[0]
    assert np.array_equal(eng.budget.cpu().numpy(), budgets)
    assert (budgets[labels == 1] > B_g).any()          # some global head gained tokens
    tr = oracle_heads(w, heads, labels, record=steps, record_pos=steps, budgets=budgets)
    worst = 0.0
    for (s, l, h) in heads:
        t_r, i = tr[(s, l, h)], flat(w, s, l, h)
        for t in steps:
            assert np.array_equal(poss[t][i], t_r.pos_at[t]), (name, s, l, h, t)
            worst = max(worst, float(np.abs(outs[t][l, s, h] - t_r.outputs[t]).max()))
        assert poss[w.n_image - 1][i].size == w.n_cond + int(budgets[i]) + t_r.nbuf
    assert worst <= TOL[w.dtype], worst
