"""hkv_decode_attention on hand-built ragged caches against the oracle's Eq. 1
(fp64), across lengths that exercise the split-K cut: empty heads, heads of
one token, heads shorter and longer than a CTA's range, many short heads, one
very long head, and a layer other than 0."""
import numpy as np
import pytest

from oracle import headkv as O

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-5, "bf16": 2e-3}


def make_cfg(H, nheads, D, dtype, n_layers=1):
    return H.make_config(n_layers=n_layers, n_seqs=1, n_heads=nheads, head_dim=D, dtype=dtype,
                         n_cond=1, n_image=64, row_len=8, recent_w=8, local_w=8, period=8,
                         group_at=8, global_budget=16)


def run_case(lens, D, dtype, seed, n_layers=1, layer=0, repeat=2):
    import torch
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import CacheBuffers, torch_dtype
    rng = np.random.default_rng(seed)
    nh = len(lens)
    cfg = make_cfg(H, nh, D, dtype, n_layers)
    dt = torch_dtype(cfg)
    n_all = nh * n_layers
    all_lens = np.concatenate([rng.integers(0, 50, size=nh * layer), lens,
                               rng.integers(0, 50, size=nh * (n_layers - layer - 1))]).astype(np.int64)
    caps = all_lens + rng.integers(0, 5, size=n_all)
    off = np.zeros(n_all, dtype=np.int64)
    off[1:] = np.cumsum(caps)[:-1]
    total = int(caps.sum())
    cb = CacheBuffers(cfg, total, "cuda")
    Kh = (rng.normal(size=(max(total, 1), D)) * 1.0).astype(np.float32)
    Vh = rng.normal(size=(max(total, 1), D)).astype(np.float32)
    cb.k.copy_(torch.from_numpy(Kh).to(dt))
    cb.v.copy_(torch.from_numpy(Vh).to(dt))
    cb.off.copy_(torch.from_numpy(off))
    cb.cap.copy_(torch.from_numpy(caps.astype(np.int32)))
    cb.len.copy_(torch.from_numpy(all_lens.astype(np.int32)))
    q = torch.from_numpy(rng.normal(size=(nh, D)).astype(np.float32) * 2.0).to(dt).cuda()
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(repeat):
        out = torch.full((nh, D), float("nan"), dtype=torch.float32, device="cuda")
        H.hkv_decode_attention(cfg, cb.c, layer, q, out, ws, ws.numel(),
                               torch.cuda.current_stream().cuda_stream)
        outs.append(out.cpu().numpy())
    H.hkv_check(cb.c)
    # the control block after the partial slots (4 per CTA boundary and one
    # per CTA, D + 4 floats each) and the boundary records (16 bytes per CTA),
    # 4096 CTAs at most, every region 256-byte aligned: the launch passed its
    # checks (int32 at byte 0)
    a256 = lambda b: (b + 255) // 256 * 256
    pf = (D + 4) * 4
    at = a256(4096 * 4 * pf) + a256(4096 * pf) + a256(4096 * 16)
    ctl = ws[at:at + 256].view(torch.int32)
    assert int(ctl[0]) == 1
    Kx = cb.k.float().cpu().numpy().astype(np.float64)
    Vx = cb.v.float().cpu().numpy().astype(np.float64)
    qx = q.float().cpu().numpy().astype(np.float64)
    base = layer * nh
    err = 0.0
    for h in range(nh):
        o, ln = int(off[base + h]), int(all_lens[base + h])
        ref = O.attention(qx[h], Kx[o:o + ln], Vx[o:o + ln])
        err = max(err, float(np.abs(outs[0][h] - ref).max()))
    assert err <= TOL[dtype], err
    for o2 in outs[1:]:
        assert np.array_equal(o2.view(np.uint32), outs[0].view(np.uint32))   # deterministic
    return err


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("D", [64, 128])
def test_mixed_lengths(dtype, D):
    lens = np.array([0, 1, 2, 17, 63, 64, 65, 500, 3000, 1, 0, 129, 2049, 7, 1200, 333] * 3)
    run_case(lens, D, dtype, seed=D + len(dtype))


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_one_long_head(dtype):
    run_case(np.array([20000]), 128, dtype, seed=3)


def test_many_short_heads():
    rng = np.random.default_rng(5)
    run_case(rng.integers(1, 6, size=3000), 128, "bf16", seed=5)


def test_uniform_global_layer():
    run_case(np.full(256, 1200), 128, "bf16", seed=6)


def test_local_global_mix_layer_offset():
    rng = np.random.default_rng(7)
    lens = np.where(rng.random(512) < 0.5, 258 + rng.integers(1, 66, 512), 1168 + rng.integers(1, 66, 512))
    run_case(lens, 128, "bf16", seed=7, n_layers=3, layer=1)


def test_all_empty_and_single_token():
    run_case(np.array([0, 0, 0]), 64, "fp32", seed=8)
    run_case(np.array([1]), 64, "bf16", seed=9)
