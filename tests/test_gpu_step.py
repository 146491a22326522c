"""The one-launch decode step (hkv_decode_step when the layer fits its head
table) on layers whose head lengths are far from equal: a few very long
heads and many short ones, so that most CTA ranges lie far from where equal
heads would put them and the prologue reads the range's counters in a
second round. Every output against Eq. 1 (the oracle's fp64 attention), and
the append and counters exact."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _skewed(H, D, dtype, seed, long_len):
    import torch
    from paper_2605_20600_gb300.engine import CacheBuffers, torch_dtype
    rng = np.random.default_rng(seed)
    nh_seq, S, L = 100, 4, 2
    cfg = H.make_config(n_layers=L, n_seqs=S, n_heads=nh_seq, head_dim=D, dtype=dtype,
                        n_cond=1, n_image=4096, row_len=64, recent_w=128, local_w=8, period=8,
                        group_at=long_len + 100, global_budget=512)
    nh = S * nh_seq
    lens = rng.integers(10, 60, size=(L, nh))
    lens[:, :40] = rng.integers(long_len - 500, long_len, size=(L, 40))  # the long heads first
    lens = lens.reshape(-1)
    caps = lens + 3
    off = np.zeros_like(caps)
    off[1:] = np.cumsum(caps)[:-1]
    total = int(caps.sum())
    cb = CacheBuffers(cfg, total, "cuda")
    dt = torch_dtype(cfg)
    cb.k.copy_(torch.from_numpy(rng.normal(size=(total, D)).astype(np.float32)).to(dt))
    cb.v.copy_(torch.from_numpy(rng.normal(size=(total, D)).astype(np.float32)).to(dt))
    cb.off.copy_(torch.from_numpy(off))
    cb.cap.copy_(torch.from_numpy(caps.astype(np.int32)))
    cb.len.copy_(torch.from_numpy(lens.astype(np.int32)))
    cb.ntok.copy_(torch.from_numpy(rng.integers(100, 200, size=L * nh).astype(np.int32)))
    return cfg, cb, rng, nh


@pytest.mark.parametrize("D,dtype,tol,long_len", [(128, "bf16", 2e-3, 3000), (64, "bf16", 2e-3, 3000),
                                                  (128, "fp32", 1e-5, 1500)])
def test_skewed_lengths_one_launch(D, dtype, tol, long_len):
    import torch
    from oracle import headkv as O
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import torch_dtype
    cfg, cb, rng, nh = _skewed(H, D, dtype, D + len(dtype), long_len)
    assert H.hkv_decode_step_launches(cfg) == 1
    dt = torch_dtype(cfg)
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    K0 = cb.k.float().cpu().numpy()
    V0 = cb.v.float().cpu().numpy()
    off = cb.off.cpu().numpy()
    for step, layer in enumerate((1, 0, 1)):   # two calls on one layer: the barrier word again
        ln0 = cb.len.cpu().numpy()
        nt0 = cb.ntok.cpu().numpy()
        q, k, v = (torch.from_numpy(rng.normal(size=(cfg.n_seqs, cfg.n_heads, D)).astype(np.float32))
                   .to(dt).cuda() for _ in range(3))
        out = torch.full((cfg.n_seqs, cfg.n_heads, D), float("nan"), dtype=torch.float32, device="cuda")
        H.hkv_decode_step(cfg, cb.c, layer, q, k, v, out, ws, ws.numel(), 0, st)
        torch.cuda.synchronize()
        H.hkv_check(cb.c)
        ln1 = cb.len.cpu().numpy()
        sl = np.arange(layer * nh, (layer + 1) * nh)
        assert (ln1[sl] == ln0[sl] + 1).all()
        assert (np.delete(ln1, sl) == np.delete(ln0, sl)).all()
        assert (cb.ntok.cpu().numpy()[sl] == nt0[sl] + 1).all()
        qn, kn, vn = (x.float().cpu().numpy().reshape(nh, D) for x in (q, k, v))
        got = out.cpu().numpy().reshape(nh, D)
        Kc = cb.k.float().cpu().numpy()
        Vc = cb.v.float().cpu().numpy()
        pos = cb.pos.cpu().numpy()
        for h in range(nh):
            i = layer * nh + h
            o, n_ = int(off[i]), int(ln0[i])
            assert np.array_equal(Kc[o + n_], kn[h]) and np.array_equal(Vc[o + n_], vn[h])
            assert pos[o + n_] == cfg.n_cond + nt0[i]
            Kh = np.vstack([K0[o:o + n_], kn[h]]) if step < 2 else Kc[o:o + n_ + 1]
            Vh = np.vstack([V0[o:o + n_], vn[h]]) if step < 2 else Vc[o:o + n_ + 1]
            exp = O.attention(qn[h], Kh, Vh)
            assert np.abs(got[h] - exp).max() <= tol, (layer, h)


@pytest.mark.parametrize("name", ["lumina1024", "llamagen_xl"])
def test_update_of_every_layer_in_one_launch_equals_one_per_layer(name):
    """hkv_evict_all runs the same update as hkv_evict on every layer: two
    engines fed the same tokens up to a due update, one updated layer by
    layer and one in one launch, hold the same cache bit for bit."""
    import torch
    from fractions import Fraction
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    from paper_2605_20600_gb300.runner import generate
    from synth import configs
    from synth.gpu import DeviceSynth
    from _gpu_util import cfg_of
    w = configs.ALL[name].with_(n_layers=3, n_seqs=2, rho=Fraction(1, 6))
    t = w.group_at + 2 * w.period      # the second update after grouping is due
    engines = []
    for per_layer in (True, False):
        eng = Engine(cfg_of(H, w), "cuda")
        generate(eng, DeviceSynth(w, "cuda"), last_step=t - 1)
        eng.release_dense()
        assert eng.update_due(t)
        nbuf0 = eng.cache.nbuf.clone()
        if per_layer:
            for layer in range(w.n_layers):
                eng.evict(layer)
        else:
            eng.evict_all()
        torch.cuda.synchronize()
        eng.check()
        engines.append((eng, nbuf0))
    (a, nb_a), (b, nb_b) = engines
    assert torch.equal(nb_a, nb_b) and int((nb_a == w.period).sum()) > 0
    for nm in ("len", "nbuf", "ntok", "off", "cap", "label"):
        assert torch.equal(getattr(a.cache, nm), getattr(b.cache, nm)), nm
    # every retained row, position and buffered query
    ln = a.cache.len.cpu().numpy()
    off = a.cache.off.cpu().numpy()
    for i in range(len(ln)):
        o, n = int(off[i]), int(ln[i])
        assert torch.equal(a.cache.k[o:o + n], b.cache.k[o:o + n]), i
        assert torch.equal(a.cache.v[o:o + n], b.cache.v[o:o + n]), i
        assert torch.equal(a.cache.pos[o:o + n], b.cache.pos[o:o + n]), i


@pytest.mark.parametrize("D,dtype,tol", [(128, "bf16", 2e-3), (64, "bf16", 2e-3), (128, "fp32", 1e-5),
                                         (64, "fp32", 1e-5)])
def test_lengths_at_tile_boundaries(D, dtype, tol):
    """Empty heads (the new token only) and lengths one below, at and one
    above every tile size the step uses (24, 48, 64 and 128 rows, by head
    dimension and type), many heads per layer, one launch: every output
    against Eq. 1, the appends and counters exact."""
    import torch
    from oracle import headkv as O
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import CacheBuffers, torch_dtype
    rng = np.random.default_rng(31 + D)
    base = [0, 1, 23, 24, 25, 47, 48, 49, 63, 64, 65, 127, 128, 129, 255, 256, 257]
    S, nh_seq, L = 3, 68, 2
    cfg = H.make_config(n_layers=L, n_seqs=S, n_heads=nh_seq, head_dim=D, dtype=dtype,
                        n_cond=1, n_image=512, row_len=16, recent_w=32, local_w=8, period=8,
                        group_at=300, global_budget=128)
    nh = S * nh_seq
    lens = np.array([base[(i * 7) % len(base)] for i in range(L * nh)], dtype=np.int64)
    caps = lens + 2
    off = np.zeros_like(caps)
    off[1:] = np.cumsum(caps)[:-1]
    total = int(caps.sum())
    cb = CacheBuffers(cfg, total, "cuda")
    dt = torch_dtype(cfg)
    cb.k.copy_(torch.from_numpy(rng.normal(size=(total, D)).astype(np.float32)).to(dt))
    cb.v.copy_(torch.from_numpy(rng.normal(size=(total, D)).astype(np.float32)).to(dt))
    cb.off.copy_(torch.from_numpy(off))
    cb.cap.copy_(torch.from_numpy(caps.astype(np.int32)))
    cb.len.copy_(torch.from_numpy(lens.astype(np.int32)))
    assert H.hkv_decode_step_launches(cfg) == 1
    K0 = cb.k.float().cpu().numpy()
    V0 = cb.v.float().cpu().numpy()
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    layer = 1
    q, k, v = (torch.from_numpy(rng.normal(size=(S, nh_seq, D)).astype(np.float32)).to(dt).cuda()
               for _ in range(3))
    out = torch.full((S, nh_seq, D), float("nan"), dtype=torch.float32, device="cuda")
    H.hkv_decode_step(cfg, cb.c, layer, q, k, v, out, ws, ws.numel(), 0, st)
    torch.cuda.synchronize()
    H.hkv_check(cb.c)
    ln1 = cb.len.cpu().numpy()
    qn, kn, vn = (x.float().cpu().numpy().reshape(nh, D) for x in (q, k, v))
    got = out.cpu().numpy().reshape(nh, D)
    Kc = cb.k.float().cpu().numpy()
    Vc = cb.v.float().cpu().numpy()
    for h in range(nh):
        i = layer * nh + h
        o, n_ = int(off[i]), int(lens[i])
        assert ln1[i] == n_ + 1
        assert np.array_equal(Kc[o + n_], kn[h]) and np.array_equal(Vc[o + n_], vn[h])
        exp = O.attention(qn[h], np.vstack([K0[o:o + n_], kn[h]]), np.vstack([V0[o:o + n_], vn[h]]))
        assert np.abs(got[h] - exp).max() <= tol, (h, n_)
    assert (ln1[:nh] == lens[:nh]).all()          # the other layer untouched
