"""A bounded device wait that runs out (failure detection without a GPU
fault). A test build of the library (-D HKV_STEP_TEST_STALL) makes the
one-launch decode step's merge warp wait for partial results of a launch
epoch that no launch writes, with the wait limit shortened to 50 ms
(-D HKV_WAIT_TIMEOUT_NS): the wait polls global memory, no bulk copy is in
flight, and the kernel must end with HKV_ERR_TIMEOUT in the cache's error
word, leaving the context usable."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def _stall_main(lib_path):
    import numpy as np
    import torch
    sys.path.insert(0, ROOT)
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    H.LIB_PATH = lib_path
    # one layer of 8 heads whose 200 conditioning tokens span several tiles,
    # so heads are split between CTAs and some CTA combines one
    cfg = H.make_config(n_layers=1, n_seqs=1, n_heads=8, head_dim=64, dtype="fp32", n_cond=200,
                        n_image=64, row_len=8, recent_w=16, local_w=16, period=8, group_at=16,
                        global_budget=32)
    assert H.hkv_decode_step_launches(cfg) == 1
    eng = Engine(cfg, "cuda")
    g = torch.Generator().manual_seed(0)
    kc = torch.randn(1, 8, 200, 64, generator=g).cuda()
    vc = torch.randn(1, 8, 200, 64, generator=g).cuda()
    eng.prefill(0, kc, vc)
    q, k, v = (torch.randn(1, 8, 64, generator=g).cuda() for _ in range(3))
    out = torch.zeros(1, 8, 64, device="cuda")
    eng.step(0, q, k, v, out)
    with pytest.raises(H.HkvError) as e:
        eng.check()
    assert e.value.status == H.HKV_ERR_TIMEOUT
    # the context is still usable
    x = torch.arange(1000, device="cuda", dtype=torch.float32)
    assert float(x.sum().item()) == 499500.0
    print("timeout ok")


def test_bounded_wait_runs_out_and_reports_timeout(tmp_path):
    sys.path.insert(0, ROOT)
    from paper_2605_20600_gb300 import build as B
    lib = str(tmp_path / "libheadkv_stall.so")
    B.build(force=True, extra_flags=["-DHKV_STEP_TEST_STALL", "-DHKV_WAIT_TIMEOUT_NS=50000000ull"],
            lib_path=lib, build_dir=str(tmp_path / "obj"))
    code = (f"import sys; sys.path.insert(0, {ROOT!r}); sys.path.insert(0, {HERE!r}); "
            f"import test_gpu_timeout as t; t._stall_main({lib!r})")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "timeout ok" in r.stdout
