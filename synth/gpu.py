"""ctypes binding of synth_gpu.cu, the GPU twin of synth/gen.py."""
from __future__ import annotations

import ctypes
import os
from ctypes import c_float, c_int, c_uint64, c_void_p

import numpy as np

from . import gen
from .configs import BF16, Workload

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libhkv_synth.so")
_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        l = ctypes.CDLL(LIB_PATH)
        l.hkv_synth_image.argtypes = [c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p,
                                      c_uint64, c_int, c_int, c_int, c_int, c_int, c_int, c_int,
                                      c_int, c_int, c_int, c_int, c_float, c_float, c_void_p]
        l.hkv_synth_image.restype = c_int
        l.hkv_synth_cond.argtypes = [c_void_p, c_void_p, c_int, c_uint64, c_int, c_int, c_int,
                                     c_int, c_int, c_float, c_float, c_void_p]
        l.hkv_synth_cond.restype = c_int
        _lib = l
    return _lib


class DeviceSynth:
    """Writes workload inputs straight into device tensors (torch)."""

    def __init__(self, w: Workload, device="cuda"):
        import torch
        self.w = w
        self.pe = torch.from_numpy(gen.pe_table(w)).to(device)
        self.cq = torch.from_numpy(gen.q_coef(w)).to(device)
        self.bf16 = 1 if w.dtype == BF16 else 0

    def image(self, q, k, v, l0: int, nl: int, t0: int, nt: int, stream: int = 0) -> None:
        """q/k/v[nt][nl][S][H][D] for image tokens t0.. and layers l0.."""
        w = self.w
        st = lib().hkv_synth_image(q.data_ptr(), k.data_ptr(), v.data_ptr(), self.bf16,
                                   self.pe.data_ptr(), self.cq.data_ptr(), w.seed, w.n_seqs,
                                   w.n_heads, w.head_dim, w.n_cond, w.row_len, w.n_image,
                                   w.n_layers, l0, nl, t0, nt, float(gen.KS), float(gen.VS),
                                   stream)
        if st != 0:
            raise RuntimeError(f"hkv_synth_image failed ({st})")

    def cond(self, kc, vc, l: int, stream: int = 0) -> None:
        """kc/vc[S][H][C][D] for layer l."""
        w = self.w
        st = lib().hkv_synth_cond(kc.data_ptr(), vc.data_ptr(), self.bf16, w.seed, w.n_seqs,
                                  w.n_heads, w.head_dim, w.n_cond, l, float(gen.KS),
                                  float(gen.VS), stream)
        if st != 0:
            raise RuntimeError(f"hkv_synth_cond failed ({st})")
