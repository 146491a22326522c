"""Schedule driver over the HeadKV C-ABI.

Owns the device buffers (allocated with torch, which serves only as the
memory and stream provider) and sequences the calls of one image generation
(Sec. 4): Step 1 cache prefilling into an uncompressed cache, Step 2 head
grouping at image token E-1, Step 3 head-aware compression (budgets, arena
allocation, repack), then decode steps of append/evict + attention. All
compute runs in libheadkv.so kernels.
"""
from __future__ import annotations

import torch

from . import hkv as H

_TORCH_DTYPE = {H.HKV_FP32: torch.float32, H.HKV_BF16: torch.bfloat16}


def torch_dtype(cfg: H.hkv_config) -> torch.dtype:
    return _TORCH_DTYPE[cfg.dtype]


class CacheBuffers:
    """Device buffers behind one hkv_cache (layout documented in hkv.h)."""

    def __init__(self, cfg: H.hkv_config, capacity_tokens: int, device, *, qbuf=None, label=None,
                 off=None, cap=None):
        n = cfg.n_layers * cfg.n_seqs * cfg.n_heads
        D, dt = cfg.head_dim, torch_dtype(cfg)
        self.k = torch.empty(max(capacity_tokens, 1), D, dtype=dt, device=device)
        self.v = torch.empty(max(capacity_tokens, 1), D, dtype=dt, device=device)
        self.pos = torch.full((max(capacity_tokens, 1),), -1, dtype=torch.int32, device=device)
        self.off = off if off is not None else torch.zeros(n, dtype=torch.int64, device=device)
        self.cap = cap if cap is not None else torch.zeros(n, dtype=torch.int32, device=device)
        self.len = torch.zeros(n, dtype=torch.int32, device=device)
        self.nbuf = torch.zeros(n, dtype=torch.int32, device=device)
        self.ntok = torch.zeros(n, dtype=torch.int32, device=device)
        self.label = label if label is not None else torch.full((n,), H.HKV_DENSE, dtype=torch.uint8,
                                                                 device=device)
        self.qbuf = qbuf if qbuf is not None else torch.zeros(n, cfg.period, D, dtype=dt, device=device)
        self.err = torch.zeros(1, dtype=torch.int32, device=device)
        self.capacity_tokens = capacity_tokens
        self.c = H.hkv_cache(self.k.data_ptr(), self.v.data_ptr(), self.pos.data_ptr(),
                             self.off.data_ptr(), self.cap.data_ptr(), self.len.data_ptr(),
                             self.nbuf.data_ptr(), self.ntok.data_ptr(), self.label.data_ptr(),
                             self.qbuf.data_ptr(), self.err.data_ptr(), capacity_tokens)


class Engine:
    """One batch of sequences through the HeadKV decode path."""

    def __init__(self, cfg: H.hkv_config, device="cuda"):
        H.hkv_validate_config(cfg)
        self.cfg = cfg
        self.device = torch.device(device)
        self.n = cfg.n_layers * cfg.n_seqs * cfg.n_heads
        seg = cfg.n_cond + cfg.group_at
        self.dense = CacheBuffers(cfg, self.n * seg, self.device)
        self.labels = torch.full((self.n,), H.HKV_DENSE, dtype=torch.uint8, device=self.device)
        self.n_h = torch.zeros(self.n, dtype=torch.int32, device=self.device)
        self.ws_bytes = H.hkv_workspace_size(cfg)
        self.ws = torch.zeros(self.ws_bytes, dtype=torch.uint8, device=self.device)
        self.ragged: CacheBuffers | None = None
        self.budget = self.cap = self.off = None
        self.total_tokens = 0
        H.hkv_init_dense(cfg, self.dense.c, self.stream())
        self.cache = self.dense

    @staticmethod
    def stream() -> int:
        return torch.cuda.current_stream().cuda_stream

    # Step 1
    def prefill(self, layer: int, kc, vc) -> None:
        H.hkv_prefill(self.cfg, self.dense.c, layer, kc, vc, self.stream())

    # per decode step and layer
    def append(self, layer: int, q, k, v) -> None:
        H.hkv_append_evict(self.cfg, self.cache.c, layer, q, k, v, self.stream())

    def attend(self, layer: int, q, out) -> None:
        H.hkv_decode_attention(self.cfg, self.cache.c, layer, q, out, self.ws, self.ws_bytes,
                               self.stream())

    # fused path: the update when due, then append + attention in one launch
    def evict(self, layer: int) -> None:
        H.hkv_evict(self.cfg, self.cache.c, layer, self.stream())

    def evict_all(self) -> None:
        """The periodic update of every layer in one launch."""
        H.hkv_evict_all(self.cfg, self.cache.c, self.stream())

    def step(self, layer: int, q, k, v, out) -> None:
        # layers run in order, so with two or more layers the kernel before a
        # decode step belongs to another layer (or is hkv_evict, which never
        # lets its successor start early): the step may prefetch
        flags = H.HKV_STEP_PREFETCH if self.cfg.n_layers >= 2 else 0
        H.hkv_decode_step(self.cfg, self.cache.c, layer, q, k, v, out, self.ws, self.ws_bytes,
                          flags, self.stream())

    def update_due(self, t: int) -> bool:
        """Whether image token t's step starts with the periodic update
        (decided by the library, hkv_update_due)."""
        return H.hkv_update_due(self.cfg, t)

    # Step 2
    def step_identify(self, layer: int, q, k, v, out) -> None:
        """The decode step of the grouping token with the head types (Sec. 4,
        Step 2) decided in the same pass, into self.labels (no n_h)."""
        flags = H.HKV_STEP_PREFETCH if self.cfg.n_layers >= 2 else 0
        H.hkv_decode_step_identify(self.cfg, self.cache.c, layer, q, k, v, out, self.labels, self.ws,
                                   self.ws_bytes, flags, self.stream())

    def identify(self, layer: int, q) -> None:
        H.hkv_identify_heads(self.cfg, self.dense.c, layer, q, self.labels, self.n_h, self.stream())

    def identify_multi(self, layer: int) -> None:
        """Step 2 from the ring's recent queries (a variant the paper does not
        have): labels and n_h."""
        H.hkv_identify_heads_multi(self.cfg, self.dense.c, layer, self.labels, self.n_h, self.stream())

    # Step 3: budgets, arena, repack of every layer
    def compress(self, labels=None) -> None:
        if labels is not None:
            self.labels.copy_(labels)
        dev = self.device
        self.budget = torch.empty(self.n, dtype=torch.int32, device=dev)
        self.cap = torch.empty(self.n, dtype=torch.int32, device=dev)
        self.off = torch.empty(self.n, dtype=torch.int64, device=dev)
        self.total_tokens = H.hkv_allocate_budgets(self.cfg, self.labels, self.budget, self.cap,
                                                   self.off, self.stream())
        self.ragged = CacheBuffers(self.cfg, self.total_tokens, dev, qbuf=self.dense.qbuf,
                                   label=self.labels, off=self.off, cap=self.cap)
        for layer in range(self.cfg.n_layers):
            H.hkv_repack(self.cfg, self.dense.c, self.ragged.c, layer, self.stream())
        self.cache = self.ragged

    def release_dense(self) -> None:
        """Frees the uncompressed arena once the ragged cache holds everything."""
        self.dense.k = self.dense.v = self.dense.pos = None

    def check(self) -> None:
        H.hkv_check(self.cache.c, self.stream())
        if self.cache is not self.dense:
            H.hkv_check(self.dense.c, self.stream())
