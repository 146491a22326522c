"""hkv_decode_attention_noalloc, the variant for callers that cannot allocate
device memory (a C host program without a device allocator, a plugin whose
host framework owns all device memory): its scratch is a fixed array inside
the library instead of a caller-provided workspace. It must give the same
outputs as hkv_decode_attention, call after call: bit for bit when both run
the same grid, and Eq. 1 (the oracle's fp64 attention) within the stated
tolerance whatever the grid.

This file is named so that pytest collects it last."""
import ctypes
import os
import subprocess
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


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
    return cfg, cb, q, off, all_lens


def _oracle_rows(cb, q, off, lens, layer, nh):
    """Eq. 1 in fp64 (the oracle) on the device's rounded inputs."""
    from oracle import headkv as O
    K = cb.k.float().cpu().numpy()
    V = cb.v.float().cpu().numpy()
    Q = q.float().cpu().numpy()
    rows = []
    for h in range(nh):
        i = layer * nh + h
        o, n = int(off[i]), int(lens[i])
        rows.append(O.attention(Q[h], K[o:o + n], V[o:o + n]))
    return np.stack(rows)


@pytest.mark.parametrize("dtype,tol", [("bf16", 2e-3), ("fp32", 1e-5)])
def test_matches_workspace_version_two_calls_in_a_row(dtype, tol):
    import torch
    from paper_2605_20600_gb300 import hkv as H
    lens = [0, 1, 5, 64, 65, 300, 1233, 323, 2000, 17] * 6
    cfg, cb, q, off, all_lens = _ragged_cache(H, lens, 128, dtype, seed=11)
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
        # the partial area holds the grid hkv_decode_attention uses here (one
        # grid per device and shape): the same kernels on the same split
        assert torch.equal(out, ref), (layer, (out - ref).abs().max().item())
        exp = _oracle_rows(cb, q, off, all_lens, layer, len(lens))
        assert np.abs(out.cpu().numpy() - exp).max() <= tol


def test_seventy_thousand_heads_match_workspace_version():
    # the scratch array has no per-head part: any number of heads fits
    import torch
    from paper_2605_20600_gb300 import hkv as H
    rng = np.random.default_rng(13)
    lens = rng.integers(0, 4, size=70000)
    cfg, cb, q, off, all_lens = _ragged_cache(H, lens, 64, "bf16", seed=13)
    st = torch.cuda.current_stream().cuda_stream
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    ref = torch.zeros(len(lens), 64, dtype=torch.float32, device="cuda")
    H.hkv_decode_attention(cfg, cb.c, 1, q, ref, ws, ws.numel(), st)
    out = torch.full_like(ref, float("nan"))
    assert _noalloc(H)(ctypes.byref(cfg), ctypes.byref(cb.c), 1, q.data_ptr(), out.data_ptr(),
                       st) == 0
    torch.cuda.synchronize()
    H.hkv_check(cb.c)
    assert torch.equal(out, ref)
    assert (out[torch.from_numpy(lens == 0).cuda()] == 0).all()
    sel = rng.choice(len(lens), size=400, replace=False)
    exp = _oracle_rows(cb, q, off, all_lens, 1, len(lens))
    assert np.abs(out.cpu().numpy()[sel] - exp[sel]).max() <= 2e-3


def _reduced_grid_main(lib_path):
    """Run in a child process against a library whose fixed partial area is
    64 KiB, so the entry point shrinks its grid to what the area holds."""
    import torch
    from paper_2605_20600_gb300 import hkv as H
    H.LIB_PATH = lib_path
    lens = [0, 3, 40, 500, 1233, 2000, 77] * 5
    for dtype, tol, D in (("bf16", 2e-3, 128), ("fp32", 1e-5, 64)):
        cfg, cb, q, off, all_lens = _ragged_cache(H, lens, D, dtype, seed=17)
        st = torch.cuda.current_stream().cuda_stream
        for layer in (0, 1):
            out = torch.full((len(lens), D), float("nan"), dtype=torch.float32, device="cuda")
            assert _noalloc(H)(ctypes.byref(cfg), ctypes.byref(cb.c), layer, q.data_ptr(),
                               out.data_ptr(), st) == 0
            torch.cuda.synchronize()
            H.hkv_check(cb.c)
            exp = _oracle_rows(cb, q, off, all_lens, layer, len(lens))
            err = np.abs(out.cpu().numpy() - exp).max()
            assert err <= tol, (dtype, layer, err)
    print("reduced grid ok")


def test_reduced_grid_when_the_partial_area_is_small(tmp_path):
    """The branch that shrinks the grid to fit the partial area: a test build
    of the library with a 64 KiB area (-D HKV_NOALLOC_PART_BYTES), checked
    against Eq. 1 in a child process."""
    sys.path.insert(0, os.path.dirname(HERE))
    from paper_2605_20600_gb300 import build as B
    B.build()
    obj = str(tmp_path / "hkv_noalloc.o")
    lib = str(tmp_path / "libheadkv_small.so")
    cc = B.nvcc()
    subprocess.check_call([cc, *B.ARCH, *B.FLAGS, "-DHKV_NOALLOC_PART_BYTES=65536", "-c",
                           os.path.join(B.CSRC, "hkv_noalloc.cu"), "-o", obj])
    others = [os.path.join(B.BUILD, s.replace(".cu", ".o")) for s in B.SOURCES
              if s != "hkv_noalloc.cu"]
    subprocess.check_call([cc, *B.ARCH, "-shared", *others, obj, "-o", lib])
    code = (f"import sys; sys.path.insert(0, {os.path.dirname(HERE)!r}); "
            f"sys.path.insert(0, {HERE!r}); import test_zz_no_alloc as t; "
            f"t._reduced_grid_main({lib!r})")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "reduced grid ok" in r.stdout
