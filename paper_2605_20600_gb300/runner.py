"""Drives one full image generation through the Engine (Sec. 4 Steps 1-3 and
the decode loop), taking per-step inputs from a provider object with

    provider.cond(kc, vc, layer, stream)                 # kc/vc [S][H][C][D]
    provider.image(q, k, v, l0, nl, t0, nt, stream)     # [nt][nl][S][H][D]

and handing each step's attention outputs to an optional callback.
"""
from __future__ import annotations

import torch

from .engine import Engine, torch_dtype


def generate(engine: Engine, provider, *, last_step: int | None = None, on_step=None,
             before_compress=None, fused: bool = True, first_step: int = 0,
             identify: str | None = None) -> None:
    """Runs image tokens first_step..last_step (default N-1) for every layer.

    fused: hkv_evict_all (every layer in one launch) when the update is due,
    then hkv_decode_step per layer; otherwise hkv_append_evict then
    hkv_decode_attention per layer.
    on_step(t, out) receives out [L][S][H][D] (fp32, device) after step t.
    before_compress(engine) runs after grouping, before budgets and repack.
    first_step > 0 continues a generation (the prefill is skipped).
    identify: "fused" decides the head types inside the grouping token's
    decode step (fused path only; no n_h), "separate" runs
    hkv_identify_heads after it (labels and n_h), "multi" runs
    hkv_identify_heads_multi after it (the recent queries' averaged
    attention; labels and n_h). Default: fused when the path is fused and
    the distances are the raster ones.
    """
    if identify is None:   # the fused count is the raster one
        identify = "fused" if fused and engine.cfg.distance_mode == 0 else "separate"
    if identify not in ("fused", "separate", "multi") or (identify == "fused" and not fused):
        raise ValueError(f"identify={identify!r} with fused={fused}")
    if identify == "fused" and engine.cfg.distance_mode != 0:
        raise ValueError("the fused identification counts in raster order only")
    cfg = engine.cfg
    L, S, H, D, C = cfg.n_layers, cfg.n_seqs, cfg.n_heads, cfg.head_dim, cfg.n_cond
    E = cfg.group_at
    dev, dt = engine.device, torch_dtype(cfg)
    st = engine.stream()
    if C > 0 and first_step == 0:
        kc = torch.empty(S, H, C, D, dtype=dt, device=dev)
        vc = torch.empty_like(kc)
        for layer in range(L):
            provider.cond(kc, vc, layer, st)
            engine.prefill(layer, kc, vc)
    q = torch.empty(L, S, H, D, dtype=dt, device=dev)
    k, v = torch.empty_like(q), torch.empty_like(q)
    out = torch.empty(L, S, H, D, dtype=torch.float32, device=dev)
    last = cfg.n_image - 1 if last_step is None else last_step
    for t in range(first_step, last + 1):
        provider.image(q, k, v, 0, L, t, 1, st)
        due = engine.update_due(t)
        if fused and due:
            engine.evict_all()       # every layer's buffer fills at the same token
        for layer in range(L):
            if fused:
                if t == E - 1 and identify == "fused":
                    engine.step_identify(layer, q[layer], k[layer], v[layer], out[layer])
                else:
                    engine.step(layer, q[layer], k[layer], v[layer], out[layer])
            else:
                engine.append(layer, q[layer], k[layer], v[layer])
                engine.attend(layer, q[layer], out[layer])
            if t == E - 1 and identify == "separate":
                engine.identify(layer, q[layer])
            elif t == E - 1 and identify == "multi":
                engine.identify_multi(layer)
        if on_step is not None:
            on_step(t, out)
        if t == E - 1:
            if before_compress is not None:
                before_compress(engine)
            engine.compress()
