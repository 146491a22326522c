"""Throughput of the HeadKV decode hot path on GB300.

A bench "step" is one steady-state period of P decode steps of the whole
model (all L layers): every layer appends its new token and attends over its
ragged cache at each of the P steps, and runs its periodic head-aware update
(STE + in-place compaction for global heads, window slide for local ones)
once, at the start of the period. Inputs (synthetic Q/K/V of the Lumina-mGPT
1024 shape) are resident in HBM before timing; the per-step KV working set
(several GB) is far larger than L2.

  value       image tokens/s = images x P x steps / device time
  roofline    decode attention (the dominant kernel): retained K/V bytes +
              q/out bytes per launch / measured launch time, vs measured HBM
  e2e         the same metric through the C-ABI with pinned host buffers:
              each step copies its inputs in and its outputs out
  cpu_baseline the CPU oracle on a sample of heads (spawn pool), projected

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                       [--workload lumina1024] [--rho 1/4]
"""
from __future__ import annotations

import argparse
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import tempfile
import time
from fractions import Fraction

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from synth import configs  # noqa: E402

METRIC = "image tokens/s per decode step on 1 GB300; decode-attn HBM GB/s vs peak"


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def workload(args) -> configs.Workload:
    w = configs.ALL[args.workload].with_(rho=Fraction(args.rho))
    if args.seqs:
        w = w.with_(n_seqs=args.seqs)
    return w


def steady_start(w: configs.Workload) -> int:
    """First step at whose start the update trims a full global history."""
    B_g = math.floor(w.rho * w.n_image)
    h_g = B_g - w.recent_w
    hist0 = max(0, w.group_at - w.recent_w)
    k = max(1, math.ceil(max(0, h_g - hist0) / w.period) + 1)
    return w.group_at + k * w.period


def describe(w, n_steps_window):
    return (f"{w.name}: L{w.n_layers} H{w.n_heads} D{w.head_dim} {w.dtype}, {w.n_seqs} seqs, "
            f"C={w.n_cond}, {w.rows}x{w.row_len} grid (N={w.n_image}), rho={w.rho}, "
            f"w={w.recent_w}, P={w.period}, E={w.group_at}; one step = one steady-state "
            f"period of P decode steps x L layers")


# the kernel sources of each decode-step design (one launch / two kernels),
# hashed together: a committed ncu capture applies while they are unchanged
STEP_SOURCES = {1: ["hkv_step.cu", "hkv_attn_common.cuh", "hkv_device.cuh"],
                2: ["hkv_attention.cu", "hkv_attn_common.cuh", "hkv_device.cuh"]}


def sources_digest(launches: int) -> str | None:
    import hashlib
    h = hashlib.sha256()
    try:
        for f in STEP_SOURCES[launches]:
            with open(os.path.join(ROOT, "paper_2605_20600_gb300", "csrc", f), "rb") as fh:
                h.update(fh.read())
    except (OSError, KeyError):
        return None
    return h.hexdigest()


def profiled_traffic(workload, bytes_per_launch, launches=2):
    """DRAM bytes per decode step from a committed ncu summary (profiles/*.md
    with the keys capture_of, launches, sources_sha256, traffic_ratio and
    extra_bytes_per_launch): the captured kernels' DRAM traffic over their
    algorithmic bytes, scaled to this launch, plus bytes that do not scale
    with it. None without a capture of this workload and design whose kernel
    sources are the current ones."""
    import glob
    digest = sources_digest(launches)
    if digest is None:
        return None
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md"))):
        vals = {}
        try:
            for line in open(path):
                k, _, v = line.strip().partition(": ")
                vals[k] = v
            if (vals.get("capture_of") == workload and vals.get("launches") == str(launches)
                    and vals.get("sources_sha256") == digest):
                return (float(vals["traffic_ratio"]) * bytes_per_launch
                        + float(vals.get("extra_bytes_per_launch", "0")))
        except (OSError, KeyError, ValueError):
            continue
    return None


def max_over_ranks(x: float, device) -> float:
    """The job's time is the slowest rank's: every rank calls this after its
    timed region (no-op on one process)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world, images_per_rank, steps_per_period, periods, ms) -> float:
    """Whole-job image tokens/s: the tokens every rank produced over the
    slowest rank's time."""
    return world * images_per_rank * steps_per_period * periods / (ms / 1e3)


def bench_config(w, world):
    """The workload both arms report (same keys, same values)."""
    return {"workload": describe(w, w.period), "rho": str(w.rho),
            "decode_steps_per_step": w.period, "layers": w.n_layers,
            "window_start_step": steady_start(w),
            "l2": "no flush: inputs and the per-step KV working set exceed L2",
            "parallelism": "replicas" if world > 1 else "single GPU"}


# ---------------------------------------------------------------------------
# CPU oracle timing (the baseline leg; runs in spawned processes)
# ---------------------------------------------------------------------------
def _oracle_period(args):
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    from oracle import headkv as O
    from synth import gen
    w, (s, l, h), t0 = args
    hi = gen.HeadInputs(w, s, l, h)
    hp = O.HeadParams.of(w)
    # untimed: the head's cache at the start of the window
    O.run_head(hp, hi.q, hi.k, hi.v, stop_after=t0 - 1)
    tr0 = time.perf_counter()
    O.run_head(hp, hi.q, hi.k, hi.v, stop_after=t0 + w.period - 1,
               record=range(t0, t0 + w.period))
    full = time.perf_counter() - tr0
    tr1 = time.perf_counter()
    O.run_head(hp, hi.q, hi.k, hi.v, stop_after=t0 - 1)
    prefix = time.perf_counter() - tr1
    return max(full - prefix, 1e-9)


def oracle_rate(w, t0, n_heads, seed, workers):
    """Projected image tokens/s of the CPU oracle from a sample of heads: the
    oracle time of one period for each sampled head (its run up to the window
    minus its run to the window start), averaged, times all L*S*H heads
    shared by `workers` processes. Returns the rate, the mean seconds per
    head-period and the wall time of the sample."""
    import random
    rnd = random.Random(seed)
    heads = [(rnd.randrange(w.n_seqs), rnd.randrange(w.n_layers), rnd.randrange(w.n_heads))
             for _ in range(n_heads)]
    jobs = [(w, x, t0) for x in heads]
    tw = time.perf_counter()
    with mp.get_context("spawn").Pool(workers) as pool:
        secs = pool.map(_oracle_period, jobs, chunksize=1)
    wall = time.perf_counter() - tw
    per_head_period = statistics.mean(secs)
    period_s = per_head_period * w.n_head_total / workers
    images = w.n_seqs / w.cfg_rows
    return images * w.period / period_s, per_head_period, wall


def cpu_baseline(w, t0):
    """The oracle on the host's cores: one process, and one process per core
    (os.cpu_count()), each on a sample of heads for one period, projected to
    every head of the model."""
    nproc = os.cpu_count() or 1
    one, ph1, wall1 = oracle_rate(w, t0, 16, 7, 1)
    n_all = 64 * nproc
    rate, ph, wall = oracle_rate(w, t0, n_all, 8, nproc)
    return {"value": rate, "unit": "image tokens/s", "cores": nproc, "kind": "oracle",
            "nproc": nproc, "single_process": one,
            "sample": f"{n_all} random heads of {w.n_head_total} on {nproc} processes (one per "
                      f"core), one period each (P={w.period} steps incl. the update) after a "
                      f"simulated run to step {t0}: mean {ph * 1e3:.1f} ms per head-period, "
                      f"{wall:.1f} s wall; the value is projected to all heads "
                      f"(x {w.n_head_total / n_all:.0f}). One process: 16 heads, "
                      f"{ph1 * 1e3:.1f} ms per head-period, {one:.1f} image tokens/s projected"}


def run_reference(args):
    """--impl reference: the CPU oracle as the reference arm. Each step times
    the oracle on a sample of heads on every host core and projects it to the
    whole model; the line says so and gives the wall time actually spent."""
    w = workload(args)
    t0 = steady_start(w)
    nproc = os.cpu_count() or 1
    n_heads = 4 * nproc
    vals, walls = [], []
    tw = time.perf_counter()
    for j in range(args.warmup + args.steps):
        v, _, wall = oracle_rate(w, t0, n_heads, 1000 + j, nproc)
        if j >= args.warmup:
            vals.append(v)
            walls.append(wall)
    value = statistics.mean(vals)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "image tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * (w.n_seqs / w.cfg_rows) * w.period / value,
        "ms_per_step_projected": True,
        "measured_wall_s": time.perf_counter() - tw,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": bench_config(w, args.gpus),
        "cpu_baseline": {"value": value, "unit": "image tokens/s", "cores": nproc,
                         "kind": "oracle", "nproc": nproc,
                         "sample": f"per step {n_heads} random heads of {w.n_head_total}, one "
                                   f"period each after a simulated run to step {t0}, on {nproc} "
                                   f"processes; ms_per_step is projected to all heads "
                                   f"(x {w.n_head_total / n_heads:.0f}), the timed samples took "
                                   f"{statistics.mean(walls):.2f} s wall each"},
        "e2e": {"value": value, "unit": "image tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
class ClockSampler:
    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,"
                 "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
                 "clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 6 and parts[0].isdigit():
                    rows.append(parts)
        except Exception:
            pass
        finally:
            if self.path:
                os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [int(r[0]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[2 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": int(rows[0][1]), "reasons": reasons,
                "samples": len(rows)}


def measure_period(args, w, dev, world, K, W, *, e2e: bool):
    """One workload on the GPU: generation up to the steady-state window, then
    K timed periods (after W warm-up periods) replayed from a CUDA graph.
    Returns the device time, per-launch roofline figures and (e2e) the same
    metric through pinned host buffers."""
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine, torch_dtype
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth

    L, S, Hh, D, P = w.n_layers, w.n_seqs, w.n_heads, w.head_dim, w.period
    t0 = steady_start(w)
    # resident input periods (fresh inputs for every timed period while they
    # fit in the image; beyond that the pool is reused cyclically)
    n_pool = max(1, min(W + K, (w.n_image - t0) // P))
    redistribute = args.budget == "redistribute"
    grid2d = args.distance == "grid2d"
    cfg = H.make_config(n_layers=L, n_seqs=S, n_heads=Hh, head_dim=D, dtype=w.dtype,
                        n_cond=w.n_cond, n_image=w.n_image, row_len=w.row_len,
                        recent_w=w.recent_w, local_w=w.w_loc, period=P, group_at=w.group_at,
                        rho=w.rho, tau=w.tau, r_s=w.r_s,
                        budget_mode=H.HKV_BUDGET_REDISTRIBUTE if redistribute else
                        H.HKV_BUDGET_PAPER,
                        distance_mode=H.HKV_DIST_GRID2D if grid2d else H.HKV_DIST_RASTER)
    eng = Engine(cfg, dev)
    synth = DeviceSynth(w, dev)
    generate(eng, synth, last_step=t0 - 1)      # dense phase, grouping, compression, decode
    eng.release_dense()
    torch.cuda.synchronize()
    eng.check()
    labels = eng.labels.cpu().numpy()
    dt = torch_dtype(cfg)

    # resident inputs of every period of the window: [n][3][P][L][S][H][D]
    pool = torch.empty(n_pool, 3, P, L, S, Hh, D, dtype=dt, device=dev)
    for j in range(n_pool):
        synth.image(pool[j, 0], pool[j, 1], pool[j, 2], 0, L, t0 + j * P, P)
    staging = torch.empty(3, P, L, S, Hh, D, dtype=dt, device=dev)
    out = torch.empty(P, L, S, Hh, D, dtype=torch.float32, device=dev)

    per_layer = args.update == "per-layer"

    def period_calls(events=None, staging=staging, out=out):
        # the period starts with the update of every layer (every buffer is
        # full): one launch for all layers, or one before each layer's first
        # step; events (instrumented copy only): [step_begin, step_end] per
        # decode step, then [update_begin, update_end] per update launch
        for p in range(P):
            if p == 0 and not per_layer:
                if events is not None:
                    events[P * L][0].record()
                eng.evict_all()
                if events is not None:
                    events[P * L][1].record()
            for layer in range(L):
                if p == 0 and per_layer:
                    if events is not None:
                        events[P * L + layer][0].record()
                    eng.evict(layer)
                    if events is not None:
                        events[P * L + layer][1].record()
                if events is not None:
                    events[p * L + layer][0].record()
                eng.step(layer, staging[0, p, layer], staging[1, p, layer], staging[2, p, layer],
                         out[p, layer])
                if events is not None:
                    events[p * L + layer][1].record()

    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        period_calls()
    stream = torch.cuda.current_stream()
    # per period: the kernels of every decode step (one launch, or an
    # attention and a finishing kernel) and the update of every layer (one)
    step_launches = H.hkv_decode_step_launches(cfg)
    launches_per_step = step_launches * P * L + (L if per_layer else 1)

    def barrier():
        if world > 1:
            dist.barrier()

    j = 0
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clk:
        time.sleep(1.0)           # the sampler is up before the GPU gets busy
        for _ in range(W):
            staging.copy_(pool[j % n_pool], non_blocking=True)
            graph.replay()
            j += 1
        barrier()
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_push("hkv_timed")
        ev0.record(stream)
        for _ in range(K):
            staging.copy_(pool[j % n_pool], non_blocking=True)
            graph.replay()
            j += 1
        ev1.record(stream)
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        barrier()
    ms = ev0.elapsed_time(ev1)
    clocks = clk.summary()
    eng.check()
    ms = max_over_ranks(ms, dev)

    # dominant kernel: the fused decode step (append + attention). One more
    # period is replayed from a copy of the graph with an event pair around
    # every decode-step launch; bytes per launch follow from the lengths at
    # the period boundary (old rows at step p = boundary length - P + p).
    lens = eng.cache.len.cpu().numpy().reshape(L, S * Hh).astype(np.int64)
    es = 2 if cfg.dtype == 1 else 4
    per_launch = [int((lens[layer] - P + p).sum()) * D * 2 * es + S * Hh * D * (6 * es + 4)
                  for p in range(P) for layer in range(L)]
    bytes_per_launch = statistics.mean(per_launch)
    events = [(torch.cuda.Event(enable_timing=True, external=True),
               torch.cuda.Event(enable_timing=True, external=True)) for _ in range(P * L + (L if per_layer else 1))]
    igraph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(igraph):
        period_calls(events)
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0.record(stream)
    staging.copy_(pool[j % n_pool], non_blocking=True)
    c1.record(stream)
    j += 1
    torch.cuda.nvtx.range_push("hkv_instrumented")
    igraph.replay()
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    eng.check()
    step_us = [e0.elapsed_time(e1) * 1e3 for e0, e1 in events[:P * L]]
    evict_us = [e0.elapsed_time(e1) * 1e3 for e0, e1 in events[P * L:]]
    copy_us = c0.elapsed_time(c1) * 1e3
    # average decode-step launch in the timed graph: the period's device time
    # minus the updates and the input copy (timed above), per launch
    attn_us = (ms * 1e3 / K - sum(evict_us) - copy_us) / (P * L)
    res = {"ms": ms, "clocks": clocks, "labels": labels, "bytes_per_launch": bytes_per_launch,
           "per_launch": per_launch, "attn_us": attn_us, "step_us": step_us,
           "evict_us": evict_us, "copy_us": copy_us, "step_launches": step_launches,
           "launches_per_step": launches_per_step, "total_tokens": eng.total_tokens,
           "staging_bytes": staging.numel() * staging.element_size(),
           "out_bytes": out.numel() * out.element_size()}

    if e2e:
        # e2e through the C-ABI with pinned host buffers, pipelined as a
        # caller would run it: two input/output buffer sets, each with its
        # graph; while period i computes, a copy stream brings in period
        # i+1's inputs and takes out period i-1's outputs. The first input
        # copy and the last output copy are not overlapped; all copies are
        # inside the timed region.
        staging_b = torch.empty_like(staging)
        out_b = torch.empty_like(out)
        graph_b = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph_b):
            period_calls(staging=staging_b, out=out_b)
        graphs, stg, outs = (graph, graph_b), (staging, staging_b), (out, out_b)
        host_in = torch.empty(staging.shape, dtype=dt, pin_memory=True)
        host_out = [torch.empty(out.shape, dtype=torch.float32, pin_memory=True) for _ in range(2)]
        host_in.copy_(pool[0])
        copy_stream = torch.cuda.Stream()
        e2e_steps = max(2, min(K, 10))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        stg[0].copy_(host_in, non_blocking=True)
        done = None
        for i in range(e2e_steps):
            b = i % 2
            graphs[b].replay()
            prev_done, done = done, torch.cuda.Event()
            done.record(stream)
            with torch.cuda.stream(copy_stream):
                if prev_done is not None:  # period i-1 released buffer set 1-b
                    copy_stream.wait_event(prev_done)
                    host_out[1 - b].copy_(outs[1 - b], non_blocking=True)
                if i + 1 < e2e_steps:
                    stg[1 - b].copy_(host_in, non_blocking=True)
                copied = torch.cuda.Event()
                copied.record(copy_stream)
            stream.wait_event(copied)
        last = (e2e_steps - 1) % 2
        host_out[last].copy_(outs[last], non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        res["e2e_ms"] = e0.elapsed_time(e1)
        res["e2e_steps"] = e2e_steps
        eng.check()
    del eng, pool, staging, out, graph, igraph
    torch.cuda.empty_cache()
    return res


def run_ours(args):
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    w = workload(args)
    P = w.period
    t0 = steady_start(w)
    K, W = args.steps, args.warmup

    # CPU baseline first (spawned workers, rank 0, one GPU)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, t0)

    r = measure_period(args, w, dev, world, K, W, e2e=True)
    images = w.n_seqs / w.cfg_rows
    value = job_value(world, images, P, K, r["ms"])
    peak, peak_kind = load_peaks()
    achieved = r["bytes_per_launch"] / (r["attn_us"] / 1e6) / 1e9
    e2e_value = world * images * P * r["e2e_steps"] / (r["e2e_ms"] / 1e3)

    # the other budgets of the same workload (Sec. 5.1's rho): fewer periods
    sweep = {}
    spec = args.rho_sweep if args.rho_sweep is not None else (
        "1/4,1/6,1/8" if w.name == "lumina1024" and not args.seqs else "")
    for rho in [x for x in spec.split(",") if x and Fraction(x) != w.rho]:
        ws = w.with_(rho=Fraction(rho))
        ks, wk = max(3, min(K, 10)), max(3, min(W, 3))
        rs = measure_period(args, ws, dev, world, ks, wk, e2e=False)
        ach = rs["bytes_per_launch"] / (rs["attn_us"] / 1e6) / 1e9
        sweep[rho] = {"value": job_value(world, images, ws.period, ks, rs["ms"]),
                      "ms_per_step": rs["ms"] / ks, "steps": ks, "warmup": wk,
                      "achieved": ach, "frac": ach / peak, "bytes_per_launch": rs["bytes_per_launch"],
                      "launch_us": rs["attn_us"], "evict_us_per_period": sum(rs["evict_us"]),
                      "global_head_fraction": float((rs["labels"] == 1).mean()),
                      "clocks": rs["clocks"]}

    if rank == 0:
        launches = r["step_launches"]
        kernel = ("hkv_decode_step: step_kernel (one launch: attention, append, merges, counters)"
                  if launches == 1 else
                  "hkv_decode_step: attn_kernel<fused> + finish_kernel<fused>")
        line = {
            "metric": METRIC, "value": value, "unit": "image tokens/s", "n_gpus": world,
            "steps": K, "warmup": W, "ms_per_step": r["ms"] / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
            "config": {**bench_config(w, world),
                       **({"budget": "redistributed (aggregate-preserving), arena "
                                     f"{r['total_tokens']} tokens"}
                          if args.budget == "redistribute" else {}),
                       **({"distance": "grid (identification and Eq. 5 strata by squared "
                                       "distance on the image grid)"}
                          if args.distance == "grid2d" else {}),
                       "update": ("every layer in one launch (hkv_evict_all)" if args.update == "all"
                                  else "one launch per layer (hkv_evict)")},
            "global_head_fraction": float((r["labels"] == 1).mean()),
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak,
                         "traffic": profiled_traffic(w.name, r["bytes_per_launch"], launches),
                         "kernel": kernel,
                         "bytes_per_launch": r["bytes_per_launch"], "launch_us": r["attn_us"],
                         # the first step of the period, per layer (what a
                         # profiler capturing the first launches sees)
                         "bytes_first_step": r["per_launch"][:w.n_layers],
                         "launch_us_isolated": statistics.mean(r["step_us"]),
                         "evict_us_per_period": sum(r["evict_us"]),
                         "copy_us_per_period": r["copy_us"],
                         "peak_kind": peak_kind},
            "rho_sweep": sweep,
            "e2e": {"value": e2e_value, "unit": "image tokens/s",
                    "h2d_bytes_per_step": r["staging_bytes"],
                    "d2h_bytes_per_step": r["out_bytes"]},
            "gpu_launches": r["launches_per_step"] * K,
            "clocks": r["clocks"],
        }
        if cpu is not None:
            line["cpu_baseline"] = cpu
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def padded_gather(cache, o, l, width):
    """K, V [..., width, D] and the key mask [..., width] of heads at arena
    offsets o with live lengths l, as a padded layout would store them (rows
    past a head's length repeat its row 0 and are masked)."""
    import torch
    ar = torch.arange(width, device=o.device)
    mask = ar < l[..., None]
    idx = torch.where(mask, o[..., None] + ar, o[..., None])
    return cache.k[idx], cache.v[idx], mask


def strategy_padding(q, cache, off, ln, width, dtype):
    """The paper's padding strategy for heads of different lengths: every head
    padded to `width` keys and masked, one batched attention per layer
    (PyTorch's scaled_dot_product_attention, computed in `dtype`).
    q [L, n, D]; off, ln [L, n]. Returns a closure filling out [L, n, D] and
    the padded tensors' bytes read per layer."""
    import torch.nn.functional as F
    L, n, D = q.shape
    Kp, Vp, Mp = padded_gather(cache, off, ln, width)
    Kp, Vp, qd = Kp.to(dtype), Vp.to(dtype), q.to(dtype)

    def run(out):
        for layer in range(L):
            o = F.scaled_dot_product_attention(
                qd[layer].reshape(1, n, 1, D), Kp[layer].reshape(1, n, width, D),
                Vp[layer].reshape(1, n, width, D), attn_mask=Mp[layer].reshape(1, n, 1, width))
            out[layer] = o.reshape(n, D)
    return run, n * width * D * 2 * Kp.element_size()


def strategy_per_group(q, cache, off, ln, cap, lab, dtype):
    """The paper's per-group strategy: one dense batch per (layer, head
    group: local, global), each padded to its group's capacity and masked
    (scaled_dot_product_attention in `dtype`). Returns a closure filling
    out [L, n, D] and the bytes read per layer."""
    import torch.nn.functional as F
    L, n, D = q.shape
    batches = []
    for layer in range(L):
        for g in (0, 1):   # local, global
            h = (lab[layer] == g).nonzero().flatten()
            if len(h) == 0:
                continue
            width = int(cap[layer][h].max())
            Kg, Vg, Mg = padded_gather(cache, off[layer][h], ln[layer][h], width)
            batches.append((layer, h, q[layer][h].contiguous().to(dtype), Kg.to(dtype),
                            Vg.to(dtype), Mg, width))

    def run(out):
        for layer, h, qg, Kg, Vg, Mg, width in batches:
            m = len(h)
            o = F.scaled_dot_product_attention(
                qg.reshape(1, m, 1, D), Kg.reshape(1, m, width, D), Vg.reshape(1, m, width, D),
                attn_mask=Mg.reshape(1, m, 1, width))
            out[layer].index_copy_(0, h, o.reshape(m, D).to(out.dtype))
    es = batches[0][3].element_size() if batches else 2
    return run, sum(len(b[1]) * b[6] * D * 2 * es for b in batches) / L


def strategies_setup(w, dev):
    """A steady-state cache of workload w (every layer right after the
    period's update) and the next step's queries."""
    import torch
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine, torch_dtype
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth
    L, S, Hh, D, P = w.n_layers, w.n_seqs, w.n_heads, w.head_dim, w.period
    t0 = steady_start(w)
    cfg = H.make_config(n_layers=L, n_seqs=S, n_heads=Hh, head_dim=D, dtype=w.dtype,
                        n_cond=w.n_cond, n_image=w.n_image, row_len=w.row_len,
                        recent_w=w.recent_w, local_w=w.w_loc, period=P, group_at=w.group_at,
                        rho=w.rho, tau=w.tau, r_s=w.r_s)
    eng = Engine(cfg, dev)
    synth = DeviceSynth(w, dev)
    generate(eng, synth, last_step=t0 - 1)
    eng.release_dense()
    eng.evict_all()
    torch.cuda.synchronize()
    eng.check()
    q = torch.empty(1, L, S, Hh, D, dtype=torch_dtype(cfg), device=dev)
    kk, vv = torch.empty_like(q), torch.empty_like(q)
    synth.image(q, kk, vv, 0, L, t0, 1)
    n = S * Hh
    c = eng.cache
    return (eng, q[0].reshape(L, n, D), c.off.view(L, n).long(), c.len.view(L, n).long(),
            c.cap.view(L, n).long(), eng.labels.view(L, n))


def run_strategies(args):
    """--strategies: decode attention over one steady-state cache (every
    layer, right after the period's update) three ways, as the paper's
    alternatives for heads of different lengths: the ragged split-K kernel of
    this library (hkv_decode_attention), padding every head to the longest
    capacity with a key mask, and one dense batch per head group (local,
    global). The two baselines run PyTorch's scaled_dot_product_attention on
    padded tensors built once (the cache as it would be stored in that
    layout), in the cache's dtype; the outputs of all three are
    cross-checked."""
    import torch

    dev = torch.device("cuda", 0)
    w = workload(args)
    L, D, P = w.n_layers, w.head_dim, w.period
    eng, q, off, ln, cap, lab = strategies_setup(w, dev)
    n = q.shape[1]
    dt = q.dtype
    es = q.element_size()
    reps = max(3, args.steps)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]

    def timed(fn):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        ev[0].record()
        for _ in range(reps):
            fn()
        ev[1].record()
        torch.cuda.synchronize()
        return ev[0].elapsed_time(ev[1]) * 1e3 / (reps * L)   # us per layer

    out_ours = torch.empty(L, n, D, dtype=torch.float32, device=dev)

    def ours():
        for layer in range(L):
            eng.attend(layer, q[layer], out_ours[layer])

    us_ours = timed(ours)
    eng.check()
    bytes_ours = float((ln.sum() * D * 2 * es).item()) / L

    out_pad = torch.empty(L, n, D, dtype=dt, device=dev)
    pad, bytes_pad = strategy_padding(q, eng.cache, off, ln, int(cap.max()), dt)
    us_pad = timed(lambda: pad(out_pad))
    del pad
    out_grp = torch.empty(L, n, D, dtype=dt, device=dev)
    grp, bytes_grp = strategy_per_group(q, eng.cache, off, ln, cap, lab, dt)
    us_grp = timed(lambda: grp(out_grp))
    err_pad = float((out_pad.float() - out_ours).abs().max())
    err_grp = float((out_grp.float() - out_ours).abs().max())
    peak, peak_kind = load_peaks()
    line = {"strategies": describe(w, P), "unit": "us per layer (attention only)",
            "ragged_splitk": {"us": us_ours, "retained_bytes": bytes_ours,
                              "GBps": bytes_ours / us_ours / 1e3},
            "padding_mask_sdpa": {"us": us_pad, "bytes_read": bytes_pad,
                                  "GBps": bytes_pad / us_pad / 1e3, "max_abs_diff": err_pad},
            "per_group_sdpa": {"us": us_grp, "bytes_read": bytes_grp,
                               "GBps": bytes_grp / us_grp / 1e3, "max_abs_diff": err_grp},
            "peak_GBps": peak, "peak_kind": peak_kind,
            "note": "baselines: torch.nn.functional.scaled_dot_product_attention on padded "
                    "tensors (library kernels); their padded tensors are built before timing"}
    print(json.dumps(line), flush=True)


def run_phases(args):
    """--phases: the one-off kernels of one generation, each timed per launch
    with CUDA events and set against its algorithmic bytes: the conditioning
    prefill (Step 1), the grouping token's decode step with the head types
    decided in it (hkv_decode_step_identify), identification from the
    current query and from the ring's recent queries (Step 2), the budgets
    (Sec. 5.1) and the repack with its first update (Step 3). Layer 0 of
    every phase (and the single budgets call) runs inside the NVTX range
    "hkv_profiled", the profiler's target; the other layers outside it."""
    import numpy as np
    import torch

    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import CacheBuffers, Engine, torch_dtype
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth

    dev = torch.device("cuda", 0)
    w = workload(args)
    L, S, Hh, D, C, E, P = (w.n_layers, w.n_seqs, w.n_heads, w.head_dim, w.n_cond, w.group_at,
                            w.period)
    cfg = H.make_config(n_layers=L, n_seqs=S, n_heads=Hh, head_dim=D, dtype=w.dtype,
                        n_cond=C, n_image=w.n_image, row_len=w.row_len, recent_w=w.recent_w,
                        local_w=w.w_loc, period=P, group_at=E, rho=w.rho, tau=w.tau, r_s=w.r_s)
    es = 2 if cfg.dtype == 1 else 4
    n = S * Hh
    eng = Engine(cfg, dev)
    synth = DeviceSynth(w, dev)
    st = eng.stream()
    res = {}

    def timed(name, fn, calls, bytes_per_call):
        """fn(i) for i in calls, the first inside "hkv_profiled"; us per call."""
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in calls]
        torch.cuda.synchronize()
        for j, (i, (e0, e1)) in enumerate(zip(calls, evs)):
            if j == 0:
                torch.cuda.nvtx.range_push("hkv_profiled")
            e0.record()
            fn(i)
            e1.record()
            if j == 0:
                torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        us = statistics.mean(e0.elapsed_time(e1) * 1e3 for e0, e1 in evs)
        res[name] = {"calls": len(calls), "us_per_call": us, "bytes_per_call": bytes_per_call,
                     "GBps": bytes_per_call / us / 1e3}

    # Step 1: conditioning K/V of every head written into the dense cache
    # (read kc, vc; write K, V rows and positions)
    # (on an engine of its own: the generation below prefills its layers)
    if C > 0:
        pre = Engine(cfg, dev)
        kc = torch.empty(L, S, Hh, C, D, dtype=torch_dtype(cfg), device=dev)
        vc = torch.empty_like(kc)
        for l in range(L):
            synth.cond(kc[l], vc[l], l, st)
        timed("prefill", lambda l: pre.prefill(l, kc[l], vc[l]), range(L), n * C * (4 * D * es + 4))
        pre.check()
        del pre, kc, vc
        torch.cuda.empty_cache()
    generate(eng, synth, first_step=0, last_step=E - 2)    # the dense phase up to E - 2
    q = torch.empty(L, S, Hh, D, dtype=torch_dtype(cfg), device=dev)
    k, v = torch.empty_like(q), torch.empty_like(q)
    synth.image(q, k, v, 0, L, E - 1, 1)
    out = torch.empty(L, S, Hh, D, dtype=torch.float32, device=dev)
    # the grouping token's step: a decode step over every head's C + E - 1
    # dense rows (+ the new one), the head types decided in the same pass
    step_bytes = n * (C + E - 1) * D * 2 * es + n * D * (6 * es + 4)
    timed("grouping_step_identify",
          lambda l: eng.step_identify(l, q[l], k[l], v[l], out[l]), range(L), step_bytes)
    # Step 2 on the cache as it stands after that step (C + E rows): the keys
    # once and the query; the multi-query variant also reads min(P, E)
    # queries of the ring
    timed("identify", lambda l: eng.identify(l, q[l]), range(L), n * (C + E + 1) * D * es)
    pe = min(P, E)
    timed("identify_multi", lambda l: eng.identify_multi(l), range(L), n * (C + E + pe) * D * es)
    eng.check()
    labels = eng.labels.clone()
    # Sec. 5.1: labels in, budget, cap, off out (1 + 4 + 4 + 8 bytes a head)
    nt = L * n
    budget = torch.empty(nt, dtype=torch.int32, device=dev)
    cap = torch.empty(nt, dtype=torch.int32, device=dev)
    off = torch.empty(nt, dtype=torch.int64, device=dev)
    total = [0]

    def budgets(_):
        total[0] = H.hkv_allocate_budgets(cfg, labels, budget, cap, off, st)
    timed("budgets", budgets, [0], nt * 17)
    rag = CacheBuffers(cfg, total[0], dev, qbuf=eng.dense.qbuf, label=labels, off=off, cap=cap)
    timed("repack", lambda l: H.hkv_repack(cfg, eng.dense.c, rag.c, l, st), range(L), 0)
    H.hkv_check(rag.c, st)
    # repack: the kept rows read from the dense cache and written to the
    # ragged one (K and V), the history keys of global heads read for the
    # scores (E - w image tokens) and their P buffered queries
    kept = rag.len.view(L, n).long().sum(1).double().mean().item()
    glob = float((labels.view(L, n) == 1).sum(1).double().mean().item())
    rb = kept * D * es * 4 + glob * (max(0, E - w.recent_w) + P) * D * es
    res["repack"]["bytes_per_call"] = rb
    res["repack"]["GBps"] = rb / res["repack"]["us_per_call"] / 1e3
    peak, peak_kind = load_peaks()
    print(json.dumps({"phases": describe(w, P), "heads_per_layer": n,
                      "global_head_fraction": float((labels == 1).float().mean().item()),
                      "results": res, "peak_GBps": peak, "peak_kind": peak_kind}), flush=True)


def run_grouping(args):
    """--grouping: the grouping token's step (image token E - 1, every layer,
    on the uncompressed cache) with the head types decided two ways: a decode
    step followed by hkv_identify_heads (a second pass over every head's
    dense keys), or hkv_decode_step_identify (the decision taken in the
    step's own pass). Each way is one CUDA graph of the L layers, replayed
    after restoring the counters the step advances (the rows it writes are
    the same every time); the labels of the two ways are compared."""
    import torch

    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine, torch_dtype
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth

    dev = torch.device("cuda", 0)
    w = workload(args)
    L, S, Hh, D, E = w.n_layers, w.n_seqs, w.n_heads, w.head_dim, w.group_at
    cfg = H.make_config(n_layers=L, n_seqs=S, n_heads=Hh, head_dim=D, dtype=w.dtype,
                        n_cond=w.n_cond, n_image=w.n_image, row_len=w.row_len,
                        recent_w=w.recent_w, local_w=w.w_loc, period=w.period, group_at=E,
                        rho=w.rho, tau=w.tau, r_s=w.r_s)
    eng = Engine(cfg, dev)
    synth = DeviceSynth(w, dev)
    generate(eng, synth, last_step=E - 2)                   # the dense phase up to E - 2
    dt = torch_dtype(cfg)
    q = torch.empty(L, S, Hh, D, dtype=dt, device=dev)
    k, v = torch.empty_like(q), torch.empty_like(q)
    synth.image(q, k, v, 0, L, E - 1, 1)
    out = torch.empty(L, S, Hh, D, dtype=torch.float32, device=dev)
    c = eng.dense
    saved = [x.clone() for x in (c.len, c.nbuf, c.ntok)]

    def restore():
        for x, y in zip((c.len, c.nbuf, c.ntok), saved):
            x.copy_(y)

    def separate():
        for layer in range(L):
            eng.step(layer, q[layer], k[layer], v[layer], out[layer])
            eng.identify(layer, q[layer])

    def fused():
        for layer in range(L):
            eng.step_identify(layer, q[layer], k[layer], v[layer], out[layer])

    res, labels = {}, {}
    for name, fn in (("separate", separate), ("fused", fused)):
        restore()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            fn()
        times = []
        for rep in range(args.warmup + args.steps):
            restore()
            eng.labels.fill_(H.HKV_DENSE)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            g.replay()
            e1.record()
            torch.cuda.synchronize()
            if rep >= args.warmup:
                times.append(e0.elapsed_time(e1) * 1000.0)
        eng.check()
        labels[name] = eng.labels.cpu().numpy().copy()
        res[name] = {"us_per_layer": statistics.median(times) / L,
                     "global_fraction": float((labels[name] == H.HKV_GLOBAL).mean())}
    dense_bytes = (eng.dense.len.sum().item() + L * S * Hh) * D * 2 * (2 if w.dtype == "bf16" else 4)
    line = {"grouping": f"{w.name}: image token E-1 = {E - 1}, {L} layers x {S * Hh} heads",
            "unit": "us per layer (median of steps)", **res,
            "labels_differ": int((labels["separate"] != labels["fused"]).sum()),
            "dense_kv_bytes_per_step": dense_bytes,
            "note": "separate: hkv_decode_step then hkv_identify_heads; fused: "
                    "hkv_decode_step_identify; one CUDA graph of all layers each"}
    print(json.dumps(line), flush=True)


def run_labels(args):
    """--labels: how the head types of Step 2 depend on the threshold tau and
    on when the grouping is taken (an analogue, on the synthetic inputs, of
    the paper's grouping-accuracy study): the dense phase runs to a late
    step, and at the paper's grouping token E - 1 and at that late token the
    heads of every layer are identified (hkv_identify_heads) with tau in
    {0.85, 0.9, 0.95}, and at tau = 0.9 also by the multi-query variant
    (hkv_identify_heads_multi) and the grid-distance one. Reports the share
    of global heads, the agreement of the labels between the two points,
    between thresholds and between the identifications, and the device time
    of each identification over all layers."""
    import torch

    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine, torch_dtype
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth

    dev = torch.device("cuda", 0)
    w = workload(args)
    L, S, Hh, D, E, N = w.n_layers, w.n_seqs, w.n_heads, w.head_dim, w.group_at, w.n_image
    late = min(N, 4 * E)
    wl = w.with_(group_at=late)
    def mk(tau, distance=H.HKV_DIST_RASTER):
        return H.make_config(n_layers=L, n_seqs=S, n_heads=Hh, head_dim=D, dtype=w.dtype,
                             n_cond=w.n_cond, n_image=N, row_len=w.row_len, recent_w=w.recent_w,
                             local_w=w.w_loc, period=w.period, group_at=late, rho=w.rho,
                             tau=tau, r_s=w.r_s, distance_mode=distance)

    cfg = mk(w.tau)
    eng = Engine(cfg, dev)
    synth = DeviceSynth(wl, dev)
    dt = torch_dtype(cfg)
    q = torch.empty(L, S, Hh, D, dtype=dt, device=dev)
    k, v = torch.empty_like(q), torch.empty_like(q)
    n = L * S * Hh
    taus = (0.85, 0.9, 0.95)
    labels, times = {}, {}

    def on_step(t, out):
        if t not in (E - 1, late - 1):
            return
        synth.image(q, k, v, 0, L, t, 1)
        for tau in taus:
            c = mk(tau)
            lab = torch.empty(n, dtype=torch.uint8, device=dev)
            nh = torch.empty(n, dtype=torch.int32, device=dev)
            for layer in range(L):
                H.hkv_identify_heads(c, eng.dense.c, layer, q[layer], lab, nh, eng.stream())
            labels[(t, tau)] = lab.cpu().numpy()
        lab = torch.empty(n, dtype=torch.uint8, device=dev)
        nh = torch.empty(n, dtype=torch.int32, device=dev)
        for kind in ("single", "multi", "grid"):
            c = mk(w.tau, H.HKV_DIST_GRID2D if kind == "grid" else H.HKV_DIST_RASTER)
            for rep in range(3):  # the last of three repetitions is timed
                ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
                ev[0].record()
                for layer in range(L):
                    if kind == "multi":
                        H.hkv_identify_heads_multi(c, eng.dense.c, layer, lab, nh, eng.stream())
                    else:
                        H.hkv_identify_heads(c, eng.dense.c, layer, q[layer], lab, nh, eng.stream())
                ev[1].record()
            torch.cuda.synchronize()
            labels[(t, kind)] = lab.cpu().numpy()
            times[(t, kind)] = ev[0].elapsed_time(ev[1]) * 1e3 / L

    generate(eng, synth, last_step=late - 1, on_step=on_step, identify="separate")
    eng.check()
    g = lambda x: float((x == H.HKV_GLOBAL).mean())
    agree = lambda a, b: float((a == b).mean())
    line = {"labels": describe(w, w.period), "heads": n, "early_token": E - 1,
            "late_token": late - 1,
            "global_fraction": {str(tau): {"early": g(labels[(E - 1, tau)]),
                                           "late": g(labels[(late - 1, tau)])} for tau in taus},
            "early_late_agreement": {str(tau): agree(labels[(E - 1, tau)], labels[(late - 1, tau)])
                                     for tau in taus},
            "tau_agreement_early": {f"{a}-{b}": agree(labels[(E - 1, a)], labels[(E - 1, b)])
                                    for a, b in ((0.85, 0.9), (0.9, 0.95), (0.85, 0.95))},
            "multi_query": {
                "queries": w.period,
                "global_fraction": {"early": g(labels[(E - 1, "multi")]),
                                    "late": g(labels[(late - 1, "multi")])},
                "early_late_agreement": agree(labels[(E - 1, "multi")], labels[(late - 1, "multi")]),
                "agreement_with_single": {"early": agree(labels[(E - 1, "multi")], labels[(E - 1, "single")]),
                                          "late": agree(labels[(late - 1, "multi")], labels[(late - 1, "single")])},
                "us_per_layer": {"single_early": times[(E - 1, "single")],
                                 "multi_early": times[(E - 1, "multi")],
                                 "single_late": times[(late - 1, "single")],
                                 "multi_late": times[(late - 1, "multi")]}},
            "grid_distance": {
                "global_fraction": {"early": g(labels[(E - 1, "grid")]),
                                    "late": g(labels[(late - 1, "grid")])},
                "early_late_agreement": agree(labels[(E - 1, "grid")], labels[(late - 1, "grid")]),
                "agreement_with_raster": {"early": agree(labels[(E - 1, "grid")], labels[(E - 1, "single")]),
                                          "late": agree(labels[(late - 1, "grid")], labels[(late - 1, "single")])},
                "us_per_layer": {"early": times[(E - 1, "grid")], "late": times[(late - 1, "grid")]}},
            "note": "synthetic inputs (per-head query scale drawn log-uniform); the paper's "
                    "grouping accuracy is against its models' own attention maps"}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="lumina1024", choices=sorted(configs.ALL))
    ap.add_argument("--rho", default="1/4")
    ap.add_argument("--rho-sweep", default=None,
                    help="other budgets measured after the headline one (comma-separated; "
                         "default 1/4,1/6,1/8 for the Lumina-mGPT-1024 shape, else none)")
    ap.add_argument("--seqs", type=int, default=0, help="override the batch (profiling runs)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--strategies", action="store_true",
                    help="compare decode attention with the padding and per-group strategies")
    ap.add_argument("--update", default="all", choices=["all", "per-layer"],
                    help="the periodic update of every layer in one launch (hkv_evict_all) "
                         "or one launch per layer (hkv_evict)")
    ap.add_argument("--budget", default="paper", choices=["paper", "redistribute"],
                    help="budget rule: the paper's, or local heads' unused tokens to global heads")
    ap.add_argument("--distance", default="raster", choices=["raster", "grid2d"],
                    help="token distance of identification and Eq. 5: the paper's raster order, "
                         "or squared distance on the image grid (a variant; the CPU baseline "
                         "stays the raster oracle)")
    ap.add_argument("--grouping", action="store_true",
                    help="time the grouping step with identification separate and fused")
    ap.add_argument("--phases", action="store_true",
                    help="time the one-off kernels of a generation (prefill, grouping, "
                         "identification, budgets, repack)")
    ap.add_argument("--labels", action="store_true",
                    help="head-type shares and stability over tau and early/late grouping")
    args = ap.parse_args()
    if args.phases:
        run_phases(args)
        return
    if args.labels:
        run_labels(args)
        return
    if args.strategies:
        run_strategies(args)
        return
    if args.grouping:
        run_grouping(args)
        return
    if args.impl == "reference":
        if int(os.environ.get("RANK", "0")) == 0:
            run_reference(args)
        return
    run_ours(args)


if __name__ == "__main__":
    main()
