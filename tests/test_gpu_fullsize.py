"""Parity at the models' full sizes and in the launch configuration of the
benchmark.

* Full size: each model shape with all of its layers and sequences runs a
  whole generation through the C-ABI (fused decode step, prefetch across
  layers, as the benchmark launches it). A sample of heads is replayed by the
  oracle: labels (Step 2) bit-exact up to declared near-ties, retained
  positions (Eqs. 3-6) exact and attention outputs (Eq. 1) within the
  tolerance at sampled steps, and the retained budget (Sec. 5.1) exact.
* Benchmark launch configuration: one steady-state period (the update of
  every layer, then P decode steps of every layer) captured in a CUDA graph
  and replayed, as the benchmark times it, on a Lumina-1024-shaped cut of
  2 layers x 2 sequences; every head is checked against the oracle."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import headkv as O
from synth import configs

from _gpu_util import LABEL_TIE, flat, oracle_heads, run_gpu

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-5, "bf16": 2e-3}

FULL = [("lumina768", "1/4"), ("lumina1024", "1/4"), ("lumina1024", "1/6"),
        ("lumina1024", "1/8"), ("llamagen_xl", "1/6"), ("janus_pro_7b", "1/8")]


def sample_heads(w, rng, n=12):
    """n distinct (s, l, h): the first and last layer always, the rest random."""
    heads = {(0, 0, 0), (w.n_seqs - 1, w.n_layers - 1, w.n_heads - 1)}
    while len(heads) < n:
        heads.add((int(rng.integers(w.n_seqs)), int(rng.integers(w.n_layers)),
                   int(rng.integers(w.n_heads))))
    return sorted(heads)


def sampled_steps(w, rng, extra=8):
    E, P, N = w.group_at, w.period, w.n_image
    s = {0, E - 1, E, E + P - 1, E + P, N - P, N - 1}
    s |= set(rng.integers(E, N, size=extra).tolist())
    return sorted(x for x in s if 0 <= x < N)


def oracle_with_gpu_labels(w, heads, gpu_labels, steps):
    """Oracle traces; a head whose GPU label differs from the oracle's must be
    a near-tie (R19) and is then replayed with the GPU's label."""
    tr = oracle_heads(w, heads, None, record=steps, record_pos=steps)
    redo = []
    for x in heads:
        g = int(gpu_labels[flat(w, *x)])
        if tr[x].label_computed != g:
            assert tr[x].margin < LABEL_TIE, (x, tr[x].label_computed, g, tr[x].margin)
            redo.append(x)
    if redo:
        tr.update(oracle_heads(w, redo, gpu_labels, record=steps, record_pos=steps))
    return tr


@pytest.mark.parametrize("name,rho", FULL)
def test_full_size_sampled_heads(name, rho):
    w = configs.ALL[name].with_(rho=Fraction(rho))
    rng = np.random.default_rng(7)
    heads = sample_heads(w, rng)
    steps = sampled_steps(w, rng)
    outs, poss, labels, _, _ = run_gpu(w, out_steps=steps, pos_steps=steps,
                                       pos_heads=[flat(w, *x) for x in heads], out_heads=heads)
    g = float((labels == 1).mean())
    assert 0.2 < g < 0.8, g                       # both head types present
    tr = oracle_with_gpu_labels(w, heads, labels, steps)
    worst = 0.0
    for x in heads:
        t_r, i = tr[x], flat(w, *x)
        for t in steps:
            assert np.array_equal(poss[t][i], t_r.pos_at[t]), (name, x, t)
            worst = max(worst, float(np.abs(outs[t][x] - t_r.outputs[t]).max()))
        budget = O.global_budget(w.rho, w.n_image) if labels[i] == 1 else w.recent_w
        assert poss[w.n_image - 1][i].size == w.n_cond + budget + t_r.nbuf, (name, x)
    assert worst <= TOL[w.dtype], (name, worst)


def test_bench_launch_configuration_graph_period():
    import torch

    from bench import steady_start
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine, torch_dtype
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth
    from _gpu_util import cfg_of

    w = configs.LUMINA_1024.with_(n_layers=2, n_seqs=2)
    L, S, Hh, D, P = w.n_layers, w.n_seqs, w.n_heads, w.head_dim, w.period
    t0 = steady_start(w)
    eng = Engine(cfg_of(H, w), "cuda")
    synth = DeviceSynth(w, "cuda")
    generate(eng, synth, last_step=t0 - 1)
    eng.release_dense()
    assert eng.update_due(t0)
    dt = torch_dtype(eng.cfg)
    staging = torch.empty(3, P, L, S, Hh, D, dtype=dt, device="cuda")
    out = torch.full((P, L, S, Hh, D), float("nan"), dtype=torch.float32, device="cuda")
    synth.image(staging[0], staging[1], staging[2], 0, L, t0, P)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for p in range(P):
            for layer in range(L):
                if p == 0:
                    eng.evict(layer)
                eng.step(layer, staging[0, p, layer], staging[1, p, layer],
                         staging[2, p, layer], out[p, layer])
    graph.replay()
    torch.cuda.synchronize()
    eng.check()
    o = out.cpu().numpy()
    c = eng.cache
    off, ln, pos = c.off.cpu().numpy(), c.len.cpu().numpy(), c.pos.cpu().numpy()
    labels = eng.labels.cpu().numpy()
    heads = [(s, l, h) for l in range(L) for s in range(S) for h in range(Hh)]
    last = t0 + P - 1
    tr = oracle_with_gpu_labels(w, heads, labels, range(t0, t0 + P))
    worst = 0.0
    for x in heads:
        s, l, h = x
        i = flat(w, *x)
        got = np.sort(pos[int(off[i]): int(off[i]) + int(ln[i])])
        assert np.array_equal(got, tr[x].pos_at[last]), x
        for p in range(P):
            worst = max(worst, float(np.abs(o[p, l, s, h] - tr[x].outputs[t0 + p]).max()))
    assert worst <= TOL[w.dtype], worst
