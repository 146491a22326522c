"""hkv_decode_attention_noalloc, the variant for callers that cannot allocate
device memory (a C host program without a device allocator, a plugin whose
host framework owns all device memory): its scratch is a fixed array inside
the library instead of a caller-provided workspace. It must give the same
outputs as hkv_decode_attention, call after call.

This file is named so that pytest collects it last."""
import ctypes

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _noalloc(H):
    f = H.lib().hkv_decode_attention_noalloc
    f.argtypes = [ctypes.POINTER(H.hkv_config), ctypes.POINTER(H.hkv_cache), ctypes.c_int,
                  ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int
    return f


def _ragged_cache(H, lens, D, dtype, seed, n_layers=2):
    import torch
    from paper_2605_20600_gb300.engine import CacheBuffers, torch_dtype
    rng = np.random.default_rng(seed)
    nh = len(lens)
    cfg = H.make_config(n_layers=n_layers, n_seqs=1, n_heads=nh, head_dim=D, dtype=dtype,
                        n_cond=1, n_image=64, row_len=8, recent_w=8, local_w=8, period=8,
                        group_at=8, global_budget=16)
    all_lens = np.concatenate([np.asarray(lens)] * n_layers).astype(np.int64)
    caps = all_lens + 3
    off = np.zeros_like(caps)
    off[1:] = np.cumsum(caps)[:-1]
    total = int(caps.sum())
    cb = CacheBuffers(cfg, total, "cuda")
    dt = torch_dtype(cfg)
    cb.k.copy_(torch.from_numpy(rng.normal(size=(total, D)).astype(np.float32)).to(dt))
    cb.v.copy_(torch.from_numpy(rng.normal(size=(total, D)).astype(np.float32)).to(dt))
    cb.off.copy_(torch.from_numpy(off))
    cb.cap.copy_(torch.from_numpy(caps.astype(np.int32)))
    cb.len.copy_(torch.from_numpy(all_lens.astype(np.int32)))
    q = torch.from_numpy((rng.normal(size=(nh, D)) * 2).astype(np.float32)).to(dt).cuda()
    return cfg, cb, q


@pytest.mark.parametrize("dtype,tol", [("bf16", 2e-3), ("fp32", 1e-5)])
def test_matches_workspace_version_two_calls_in_a_row(dtype, tol):
    import torch
    from paper_2605_20600_gb300 import hkv as H
    lens = [0, 1, 5, 64, 65, 300, 1233, 323, 2000, 17] * 6
    cfg, cb, q = _ragged_cache(H, lens, 128, dtype, seed=11)
    f = _noalloc(H)
    st = torch.cuda.current_stream().cuda_stream
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    for layer in (1, 0):                      # two calls in a row, different layers
        ref = torch.zeros(len(lens), 128, dtype=torch.float32, device="cuda")
        H.hkv_decode_attention(cfg, cb.c, layer, q, ref, ws, ws.numel(), st)
        out = torch.full_like(ref, float("nan"))
        assert f(ctypes.byref(cfg), ctypes.byref(cb.c), layer, q.data_ptr(), out.data_ptr(), st) == 0
        torch.cuda.synchronize()
        H.hkv_check(cb.c)
        diff = (out - ref).abs().max().item()
        assert diff <= tol, (layer, diff)
        assert not torch.isnan(out).any()


def test_seventy_thousand_heads_match_workspace_version():
    # the scratch array has no per-head part: any number of heads fits
    import torch
    from paper_2605_20600_gb300 import hkv as H
    rng = np.random.default_rng(13)
    lens = rng.integers(0, 4, size=70000)
    cfg, cb, q = _ragged_cache(H, lens, 64, "bf16", seed=13)
    st = torch.cuda.current_stream().cuda_stream
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    ref = torch.zeros(len(lens), 64, dtype=torch.float32, device="cuda")
    H.hkv_decode_attention(cfg, cb.c, 1, q, ref, ws, ws.numel(), st)
    out = torch.full_like(ref, float("nan"))
    assert _noalloc(H)(ctypes.byref(cfg), ctypes.byref(cb.c), 1, q.data_ptr(), out.data_ptr(),
                       st) == 0
    torch.cuda.synchronize()
    H.hkv_check(cb.c)
    assert (out - ref).abs().max().item() <= 2e-3
    assert not torch.isnan(out).any()
    assert (out[torch.from_numpy(lens == 0).cuda()] == 0).all()
