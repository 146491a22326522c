"""ctypes binding of the HeadKV C-ABI (include/hkv.h).

Argument marshalling only: every function has the name of the C entry point
it forwards to, accepts integers (device addresses) or objects with a
`data_ptr()` method for pointer arguments, and raises HkvError on a status
other than HKV_OK. There is no fallback: if libheadkv.so is missing the
import of a function fails loudly.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, Structure, c_char_p, c_double, c_int, c_int32, c_int64, c_size_t, c_void_p
from fractions import Fraction

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libheadkv.so")

HKV_OK = 0
HKV_ERR_INVALID_ARG = 1
HKV_ERR_SHAPE = 2
HKV_ERR_CAPACITY = 3
HKV_ERR_STATE = 4
HKV_ERR_BOUNDS = 5
HKV_ERR_TIMEOUT = 6
HKV_ERR_CUDA = 7
HKV_ERR_ALIGN = 8

HKV_FP32, HKV_BF16 = 0, 1
HKV_STEP_PREFETCH = 1
HKV_LOCAL, HKV_GLOBAL, HKV_DENSE = 0, 1, 255
HKV_BUDGET_PAPER, HKV_BUDGET_REDISTRIBUTE = 0, 1
HKV_DIST_RASTER, HKV_DIST_GRID2D = 0, 1


class hkv_config(Structure):
    _fields_ = [
        ("n_layers", c_int32), ("n_seqs", c_int32), ("n_heads", c_int32), ("head_dim", c_int32),
        ("dtype", c_int32), ("n_cond", c_int32), ("n_image", c_int32), ("row_len", c_int32),
        ("recent_w", c_int32), ("local_w", c_int32), ("period", c_int32), ("group_at", c_int32),
        ("global_budget", c_int32), ("budget_mode", c_int32), ("distance_mode", c_int32),
        ("reserved", c_int32), ("tau", c_double), ("r_s", c_double),
    ]


class hkv_cache(Structure):
    _fields_ = [
        ("k", c_void_p), ("v", c_void_p), ("pos", c_void_p), ("off", c_void_p), ("cap", c_void_p),
        ("len", c_void_p), ("nbuf", c_void_p), ("ntok", c_void_p), ("label", c_void_p),
        ("qbuf", c_void_p), ("err", c_void_p), ("capacity_tokens", c_int64),
    ]


class HkvError(RuntimeError):
    def __init__(self, name: str, status: int):
        self.status = status
        super().__init__(f"hkv_{name}: {hkv_status_str(status)} ({status})")


_lib = None

# (name, argtypes, restype)
_SIGNATURES = {
    "hkv_status_str": ([c_int], c_char_p),
    "hkv_validate_config": ([POINTER(hkv_config)], c_int),
    "hkv_workspace_size": ([POINTER(hkv_config)], c_size_t),
    "hkv_init_dense": ([POINTER(hkv_config), POINTER(hkv_cache), c_void_p], c_int),
    "hkv_prefill": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p, c_void_p], c_int),
    "hkv_append_evict": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p, c_void_p,
                          c_void_p], c_int),
    "hkv_decode_attention": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p, c_void_p,
                              c_size_t, c_void_p], c_int),
    "hkv_decode_step": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p, c_void_p,
                         c_void_p, c_void_p, c_size_t, c_int, c_void_p], c_int),
    "hkv_decode_step_identify": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p,
                                  c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_int, c_void_p],
                                 c_int),
    "hkv_decode_step_launches": ([POINTER(hkv_config)], c_int),
    "hkv_global_budget": ([c_int64, c_int64, c_int32, POINTER(c_int32)], c_int),
    "hkv_update_due": ([POINTER(hkv_config), c_int32, POINTER(c_int32)], c_int),
    "hkv_evict": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p], c_int),
    "hkv_evict_all": ([POINTER(hkv_config), POINTER(hkv_cache), c_void_p], c_int),
    "hkv_identify_heads": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p, c_void_p,
                            c_void_p], c_int),
    "hkv_identify_heads_multi": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p,
                                  c_void_p], c_int),
    "hkv_allocate_budgets": ([POINTER(hkv_config), c_void_p, c_void_p, c_void_p, c_void_p,
                              POINTER(c_int64), c_void_p], c_int),
    "hkv_repack": ([POINTER(hkv_config), POINTER(hkv_cache), POINTER(hkv_cache), c_int, c_void_p], c_int),
    "hkv_check": ([POINTER(hkv_cache), c_void_p], c_int),
    "hkv_export_state": ([POINTER(hkv_config), POINTER(hkv_cache), c_int, c_void_p, c_void_p, c_void_p,
                          c_void_p, c_void_p, c_int64, POINTER(c_int64), c_void_p], c_int),
}


def lib():
    """The loaded libheadkv.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        l = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGNATURES.items():
            f = getattr(l, name)
            f.argtypes = args
            f.restype = res
        _lib = l
    return _lib


def _p(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _call(name: str, *args) -> None:
    st = getattr(lib(), "hkv_" + name)(*args)
    if st != HKV_OK:
        raise HkvError(name, st)


def hkv_status_str(status: int) -> str:
    return lib().hkv_status_str(status).decode()


def make_config(*, n_layers, n_seqs, n_heads, head_dim, dtype, n_cond, n_image, row_len,
                recent_w, local_w, period, group_at, rho=None, global_budget=None,
                tau=0.9, r_s=0.5, budget_mode=HKV_BUDGET_PAPER,
                distance_mode=HKV_DIST_RASTER) -> hkv_config:
    """Builds an hkv_config; the global budget is the library's
    hkv_global_budget(rho, N) unless given explicitly."""
    if global_budget is None:
        global_budget = hkv_global_budget(rho, n_image)
    return hkv_config(n_layers, n_seqs, n_heads, head_dim,
                      HKV_BF16 if dtype in ("bf16", HKV_BF16) else HKV_FP32,
                      n_cond, n_image, row_len, recent_w, local_w, period, group_at,
                      int(global_budget), int(budget_mode), int(distance_mode), 0, float(tau),
                      float(r_s))


def hkv_global_budget(rho, n_image: int) -> int:
    """B_g for a budget ratio rho (a Fraction, or anything Fraction takes)."""
    r = Fraction(rho)
    out = c_int32(0)
    _call("global_budget", r.numerator, r.denominator, n_image, ctypes.byref(out))
    return int(out.value)


def hkv_update_due(cfg: hkv_config, t: int) -> bool:
    """Whether image token t's decode step starts with the periodic update."""
    out = c_int32(0)
    _call("update_due", ctypes.byref(cfg), t, ctypes.byref(out))
    return bool(out.value)


def hkv_validate_config(cfg: hkv_config) -> None:
    _call("validate_config", ctypes.byref(cfg))


def hkv_workspace_size(cfg: hkv_config) -> int:
    return int(lib().hkv_workspace_size(ctypes.byref(cfg)))


def hkv_init_dense(cfg, cache, stream=0) -> None:
    _call("init_dense", ctypes.byref(cfg), ctypes.byref(cache), stream)


def hkv_prefill(cfg, cache, layer, kc, vc, stream=0) -> None:
    _call("prefill", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(kc), _p(vc), stream)


def hkv_append_evict(cfg, cache, layer, q, k, v, stream=0) -> None:
    _call("append_evict", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(q), _p(k), _p(v), stream)


def hkv_decode_attention(cfg, cache, layer, q, out, workspace, ws_bytes, stream=0) -> None:
    _call("decode_attention", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(q), _p(out),
          _p(workspace), ws_bytes, stream)


def hkv_decode_step(cfg, cache, layer, q, k, v, out, workspace, ws_bytes, flags=0,
                    stream=0) -> None:
    _call("decode_step", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(q), _p(k), _p(v), _p(out),
          _p(workspace), ws_bytes, flags, stream)


def hkv_decode_step_launches(cfg) -> int:
    """Kernel launches of one hkv_decode_step call (1 or 2) on the current
    device; raises on an invalid config."""
    n = int(lib().hkv_decode_step_launches(ctypes.byref(cfg)))
    if n <= 0:
        raise HkvError("decode_step_launches", HKV_ERR_INVALID_ARG)
    return n


def hkv_decode_step_identify(cfg, cache, layer, q, k, v, out, label_out, workspace, ws_bytes,
                             flags=0, stream=0) -> None:
    _call("decode_step_identify", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(q), _p(k), _p(v),
          _p(out), _p(label_out), _p(workspace), ws_bytes, flags, stream)


def hkv_evict(cfg, cache, layer, stream=0) -> None:
    _call("evict", ctypes.byref(cfg), ctypes.byref(cache), layer, stream)


def hkv_evict_all(cfg, cache, stream=0) -> None:
    _call("evict_all", ctypes.byref(cfg), ctypes.byref(cache), stream)


def hkv_identify_heads(cfg, cache, layer, q, label_out, nh_out=None, stream=0) -> None:
    _call("identify_heads", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(q), _p(label_out),
          _p(nh_out), stream)


def hkv_identify_heads_multi(cfg, cache, layer, label_out, nh_out=None, stream=0) -> None:
    _call("identify_heads_multi", ctypes.byref(cfg), ctypes.byref(cache), layer, _p(label_out),
          _p(nh_out), stream)


def hkv_allocate_budgets(cfg, label, budget, cap, off, stream=0) -> int:
    total = c_int64(0)
    _call("allocate_budgets", ctypes.byref(cfg), _p(label), _p(budget), _p(cap), _p(off),
          ctypes.byref(total), stream)
    return int(total.value)


def hkv_repack(cfg, dense, ragged, layer, stream=0) -> None:
    _call("repack", ctypes.byref(cfg), ctypes.byref(dense), ctypes.byref(ragged), layer, stream)


def hkv_check(cache, stream=0) -> None:
    _call("check", ctypes.byref(cache), stream)


def hkv_export_state(cfg, cache, layer, stream=0):
    """One layer's state on the host: numpy arrays label, len, nbuf, ntok
    (S*H each) and the live positions of every head, packed head after head
    (a list of arrays, one per head)."""
    import numpy as np
    n = cfg.n_seqs * cfg.n_heads
    label = np.zeros(n, np.uint8)
    ln = np.zeros(n, np.int32)
    nbuf = np.zeros(n, np.int32)
    ntok = np.zeros(n, np.int32)
    count = c_int64(0)
    _call("export_state", ctypes.byref(cfg), ctypes.byref(cache), layer, label.ctypes.data,
          ln.ctypes.data, nbuf.ctypes.data, ntok.ctypes.data, None, 0, ctypes.byref(count), stream)
    pos = np.zeros(max(int(count.value), 1), np.int32)
    _call("export_state", ctypes.byref(cfg), ctypes.byref(cache), layer, None, None, None, None,
          pos.ctypes.data, pos.size, ctypes.byref(count), stream)
    split = np.cumsum(ln)[:-1]
    return {"label": label, "len": ln, "nbuf": nbuf, "ntok": ntok,
            "pos": np.split(pos[:int(count.value)], split)}
