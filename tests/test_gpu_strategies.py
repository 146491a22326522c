"""The paper's alternative attention strategies for heads of different
lengths (padding every head and masking; one dense batch per head group),
as bench.py --strategies times them: correct programs, so that the timing
compares like with like. On a steady-state cache of a reduced model shape
their outputs, computed in fp32, match Eq. 1 (the oracle, fp64) within the
fp32 tolerance of the hot path's tests (2e-3 for bf16 inputs); computed in
the cache's bf16 (as timed), within that plus the rounding of a bf16
output."""
import os
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("name", ["janus_pro_7b", "lumina1024"])
def test_padding_and_per_group_match_eq1(name):
    import torch
    sys.path.insert(0, ROOT)
    import bench
    from oracle import headkv as O
    from synth import configs
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2)
    eng, q, off, ln, cap, lab = bench.strategies_setup(w, torch.device("cuda", 0))
    L, n, D = q.shape
    K = eng.cache.k.float().cpu().numpy()
    V = eng.cache.v.float().cpu().numpy()
    Q = q.float().cpu().numpy()
    offs, lens = off.cpu().numpy(), ln.cpu().numpy()
    exp = np.stack([np.stack([O.attention(Q[l, i], K[offs[l, i]:offs[l, i] + lens[l, i]],
                                          V[offs[l, i]:offs[l, i] + lens[l, i]])
                              for i in range(n)]) for l in range(L)])
    assert (lab.cpu().numpy() == 0).any() and (lab.cpu().numpy() == 1).any()
    for dtype, extra in ((torch.float32, 0.0), (q.dtype, 2.0 ** -7)):
        for make in ("padding", "per_group"):
            out = torch.full((L, n, D), float("nan"), dtype=dtype, device="cuda")
            if make == "padding":
                run, _ = bench.strategy_padding(q, eng.cache, off, ln, int(cap.max()), dtype)
            else:
                run, _ = bench.strategy_per_group(q, eng.cache, off, ln, cap, lab, dtype)
            run(out)
            torch.cuda.synchronize()
            got = out.float().cpu().numpy()
            # bf16 output: two units in the last place of |o| on top of the fp32 tolerance
            tol = 2e-3 + extra * np.abs(exp)
            assert np.all(np.abs(got - exp) <= tol), (make, dtype, float(np.abs(got - exp).max()))
