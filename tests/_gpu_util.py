"""Helpers of the GPU parity tests: workload -> config, one generation through
the C-ABI with snapshots, oracle runs of sampled heads in a spawn pool."""
from __future__ import annotations

import dataclasses
import multiprocessing as mp
import os

import numpy as np

from oracle import headkv as O
from synth import configs, gen


def cfg_of(H, w: configs.Workload, budget_mode=0, distance_mode=0):
    return H.make_config(n_layers=w.n_layers, n_seqs=w.n_seqs, n_heads=w.n_heads,
                         head_dim=w.head_dim, dtype=w.dtype, n_cond=w.n_cond, n_image=w.n_image,
                         row_len=w.row_len, recent_w=w.recent_w, local_w=w.w_loc,
                         period=w.period, group_at=w.group_at, rho=w.rho, tau=w.tau, r_s=w.r_s,
                         budget_mode=budget_mode, distance_mode=distance_mode)


def flat(w, s, l, h):
    return (l * w.n_seqs + s) * w.n_heads + h


def run_gpu(w, *, out_steps=(), pos_steps=(), pos_heads=(), last_step=None, fused=True,
            out_heads=None, identify="separate", budget_mode=0, distance_mode=0,
            force_labels=None):
    """One generation on the GPU. Returns outputs {t: [L,S,H,D] fp32, or
    {(s, l, h): [D]} for out_heads}, positions {t: {flat head: sorted
    positions}}, labels, n_h (None when the identification is fused into
    the grouping step, which gives no n_h) and the engine. force_labels (a
    flat array) replaces the labels after grouping, before compression."""
    import torch
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth

    eng = Engine(cfg_of(H, w, budget_mode, distance_mode), "cuda")
    out_steps, pos_steps = set(out_steps), set(pos_steps)
    outs, poss = {}, {}

    if out_heads is not None:
        sel = [torch.tensor([x[i] for x in out_heads], device="cuda") for i in (1, 0, 2)]

    def on_step(t, out):
        if t in out_steps:
            if out_heads is None:
                outs[t] = out.cpu().numpy()
            else:
                rows = out[sel[0], sel[1], sel[2]].cpu().numpy()
                outs[t] = {x: rows[j] for j, x in enumerate(out_heads)}
        if t in pos_steps:
            c = eng.cache
            off, ln = c.off.cpu().numpy(), c.len.cpu().numpy()
            allpos = c.pos
            poss[t] = {i: np.sort(allpos[int(off[i]): int(off[i]) + int(ln[i])].cpu().numpy())
                       for i in pos_heads}

    def before_compress(e):
        if force_labels is not None:
            e.labels.copy_(torch.as_tensor(np.asarray(force_labels, dtype=np.uint8), device="cuda"))

    generate(eng, DeviceSynth(w, "cuda"), on_step=on_step, last_step=last_step, fused=fused,
             identify=identify, before_compress=before_compress)
    torch.cuda.synchronize()
    eng.check()
    nh = eng.n_h.cpu().numpy() if identify in ("separate", "multi") else None
    return outs, poss, eng.labels.cpu().numpy(), nh, eng


def _oracle_job(args):
    w, s, l, h, label, record, record_pos, budget, distance = args
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    hi = gen.HeadInputs(w, s, l, h, pe, cq)
    hp = O.HeadParams.of(w, distance)
    if budget is not None and label == O.GLOBAL:   # a per-head budget (redistributed)
        hp = dataclasses.replace(hp, global_budget=budget)
    tr = O.run_head(hp, hi.q, hi.k, hi.v, label=label, record=record, record_pos=record_pos)
    return (s, l, h), tr


def oracle_heads(w, heads, labels=None, record=(), record_pos=(), budgets=None, distance=0):
    """Oracle traces of the given (s, l, h) heads; labels (flat array) are
    injected when given, and so are per-head image-token budgets (flat
    array, used for global heads). Runs in a spawn pool (safe after CUDA
    init)."""
    jobs = [(w, s, l, h, None if labels is None else int(labels[flat(w, s, l, h)]),
             tuple(record), tuple(record_pos),
             None if budgets is None else int(budgets[flat(w, s, l, h)]), distance)
            for (s, l, h) in heads]
    if len(jobs) <= 2:
        return dict(map(_oracle_job, jobs))
    n = min(len(jobs), os.cpu_count() or 1, 16)
    with mp.get_context("spawn").Pool(n) as pool:
        return dict(pool.map(_oracle_job, jobs, chunksize=1))


def label_job(args):
    """Oracle grouping for heads of one (s, l): (label, n_h, margin) per head;
    multi: from the newest min(P, E) queries (grouping_count_multi);
    distance: O.GRID2D counts outward on the grid."""
    w, s, l, heads, multi, distance = args
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    hp = O.HeadParams.of(w)
    res = []
    for h in heads:
        hi = gen.HeadInputs(w, s, l, h, pe, cq)
        t = w.group_at - 1
        K = hi.k[: w.n_cond + t + 1]
        Q = hi.q[max(0, t + 1 - w.period): t + 1]
        if multi and distance == O.GRID2D:
            n_h, cum = O.grouping_count_multi_2d(Q, K, w.tau, w.n_cond, w.row_len)
        elif multi:
            n_h, cum = O.grouping_count_multi(Q, K, w.tau)
        elif distance == O.GRID2D:
            n_h, cum = O.grouping_count_2d(hi.q[t], K, w.tau, w.n_cond, w.row_len)
        else:
            n_h, cum = O.grouping_count(hi.q[t], K, w.tau)
        res.append((O.classify(n_h, w.w_loc), n_h, O.label_margin(cum, w.tau, w.w_loc),
                    O.count_margin(cum, w.tau, n_h)))
    return (s, l), res


def oracle_labels(w, layers, seqs, multi=False, distance=0):
    jobs = [(w, s, l, tuple(range(w.n_heads)), multi, distance) for l in layers for s in seqs]
    n = min(len(jobs), os.cpu_count() or 1, 16)
    with mp.get_context("spawn").Pool(n) as pool:
        return dict(pool.map(label_job, jobs, chunksize=1))


# |fp64 mass - tau| below this: either decision is correct (the GPU sums the
# same weights in fp32; on every tested shape its rounding stays inside this
# band)
LABEL_TIE = 1e-5


def check_labels(w, gpu_labels, gpu_nh, oracle_lab, where):
    """Labels and n_h bit-exact, except the declared near-ties: a label may
    differ only where the fp64 mass of the newest w_loc-1 tokens is within
    LABEL_TIE of tau, n_h only where a cumulative mass next to the count's cut
    is. Returns the heads whose label differed."""
    ties = []
    for (s, l), res in oracle_lab.items():
        for h, (lab, n_h, margin, n_margin) in enumerate(res):
            i = flat(w, s, l, h)
            if int(gpu_labels[i]) != lab:
                assert margin < LABEL_TIE, (where, s, l, h, lab, int(gpu_labels[i]), margin)
                ties.append((s, l, h, margin))
            if gpu_nh is not None and int(gpu_nh[i]) != n_h:
                assert n_margin < LABEL_TIE, (where, s, l, h, n_h, int(gpu_nh[i]), n_margin)
    return ties
