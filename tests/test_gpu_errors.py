"""Device-side failures are reported through the error word, not by faulting:
a full segment, a segment outside the arena, a label in the wrong state."""
import numpy as np
import pytest

from synth import configs

from _gpu_util import cfg_of

pytestmark = pytest.mark.gpu


def small_engine():
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import Engine
    w = configs.TINY
    return H, Engine(cfg_of(H, w), "cuda"), w


def test_full_segment_sets_capacity():
    import torch
    H, eng, w = small_engine()
    eng.dense.cap[3] = 0                   # head 3 has no room at all
    S, Hh, D = w.n_seqs, w.n_heads, w.head_dim
    x = torch.zeros(S, Hh, D, device="cuda")
    eng.append(0, x, x, x)
    with pytest.raises(H.HkvError) as e:
        eng.check()
    assert e.value.status == H.HKV_ERR_CAPACITY
    ln = eng.dense.len.cpu().numpy()
    assert ln[3] == 0 and (np.delete(ln, 3) == 1).all()   # the others appended


def test_segment_outside_arena_sets_bounds():
    import torch
    H, eng, w = small_engine()
    eng.dense.len.fill_(5)
    eng.dense.off[2] = eng.dense.capacity_tokens          # starts past the end
    q = torch.zeros(w.n_seqs, w.n_heads, w.head_dim, device="cuda")
    out = torch.zeros(w.n_seqs, w.n_heads, w.head_dim, device="cuda")
    eng.attend(0, q, out)
    with pytest.raises(H.HkvError) as e:
        eng.check()
    assert e.value.status == H.HKV_ERR_BOUNDS


def test_budgets_reject_unlabelled_heads():
    H, eng, w = small_engine()
    with pytest.raises(H.HkvError) as e:
        eng.compress()                    # labels are still HKV_DENSE
    assert e.value.status == H.HKV_ERR_STATE


def test_prefill_twice_is_a_state_error():
    import torch
    H, eng, w = small_engine()
    kc = torch.zeros(w.n_seqs, w.n_heads, w.n_cond, w.head_dim, device="cuda")
    eng.prefill(0, kc, kc)
    eng.prefill(0, kc, kc)
    with pytest.raises(H.HkvError) as e:
        eng.check()
    assert e.value.status == H.HKV_ERR_STATE


def test_decode_step_refuses_a_due_update():
    """hkv_decode_step on a head whose buffer is full (hkv_evict skipped)
    reports a state error and takes no step; hkv_evict then unblocks it."""
    import torch
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth
    H, eng, w = small_engine()
    E, P = w.group_at, w.period
    generate(eng, DeviceSynth(w, "cuda"), last_step=E + P - 1)       # buffer now full
    eng.check()
    ln = eng.cache.len.clone()
    q = torch.zeros(w.n_seqs, w.n_heads, w.head_dim, device="cuda")
    out = torch.zeros(w.n_seqs, w.n_heads, w.head_dim, device="cuda")
    eng.step(0, q, q, q, out)
    with pytest.raises(H.HkvError) as e:
        eng.check()
    assert e.value.status == H.HKV_ERR_STATE
    assert torch.equal(eng.cache.len, ln)
    eng.cache.err.zero_()
    eng.ws.zero_()
    eng.evict(0)
    eng.step(0, q, q, q, out)
    eng.check()
    assert (eng.cache.len.cpu() <= eng.cache.cap.cpu()).all()


def test_evict_is_a_no_op_when_not_due():
    from paper_2605_20600_gb300.runner import generate
    from synth.gpu import DeviceSynth
    H, eng, w = small_engine()
    generate(eng, DeviceSynth(w, "cuda"), last_step=w.group_at + 2)
    before = (eng.cache.len.clone(), eng.cache.pos.clone(), eng.cache.k.clone())
    eng.evict(0)
    eng.check()
    assert torch_equal_all(before, (eng.cache.len, eng.cache.pos, eng.cache.k))


def torch_equal_all(a, b):
    """Bitwise equality (the arena's unused rows may hold NaN patterns left
    in recycled device memory, which compare unequal to themselves)."""
    import torch
    return all(torch.equal(x.contiguous().view(torch.uint8), y.contiguous().view(torch.uint8))
               for x, y in zip(a, b))


def _step_cache(seed, nh=96, D=128, n_layers=2):
    """A ragged bf16 cache of nh heads per layer with lengths from 20 to 700
    rows, so that the one-launch decode step splits heads across CTAs."""
    import torch
    from paper_2605_20600_gb300 import hkv as H
    from paper_2605_20600_gb300.engine import CacheBuffers, torch_dtype
    rng = np.random.default_rng(seed)
    cfg = H.make_config(n_layers=n_layers, n_seqs=1, n_heads=nh, head_dim=D, dtype="bf16",
                        n_cond=1, n_image=64, row_len=8, recent_w=8, local_w=8, period=8,
                        group_at=8, global_budget=16)
    n = n_layers * nh
    lens = rng.integers(20, 700, size=n)
    caps = lens + 4
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
    cb.label.copy_(torch.from_numpy(rng.integers(0, 2, size=n).astype(np.uint8)))
    cb.nbuf.copy_(torch.from_numpy(rng.integers(0, cfg.period, size=n).astype(np.int32)))
    cb.ntok.copy_(torch.from_numpy(rng.integers(100, 200, size=n).astype(np.int32)))
    return H, cfg, cb, rng


@pytest.mark.parametrize("head", [0, 57, 95])
@pytest.mark.parametrize("fault", ["capacity", "state", "bounds"])
def test_one_bad_head_stops_the_whole_one_launch_step(fault, head):
    """In the one-launch decode step each CTA checks only the heads of its own
    range; a bad head anywhere must still leave every head of the layer
    untouched (no append, no counter), and the next call, with the fault
    repaired, takes the step and matches Eq. 1."""
    import torch
    from oracle import headkv as O
    H, cfg, cb, rng = _step_cache(7 + head)
    assert H.hkv_decode_step_launches(cfg) == 1
    nh, D, layer = cfg.n_heads, cfg.head_dim, 1
    i = layer * nh + head
    field, good = {"capacity": (cb.cap, cb.len[i].item()),
                   "state": (cb.nbuf, cfg.period),
                   "bounds": (cb.off, cb.capacity_tokens)}[fault]
    old = field[i].item()
    if fault == "state":
        cb.label[i] = H.HKV_GLOBAL
    field[i] = good
    q, k, v = (torch.from_numpy(rng.normal(size=(1, nh, D)).astype(np.float32))
               .to(torch.bfloat16).cuda() for _ in range(3))
    out = torch.zeros(1, nh, D, dtype=torch.float32, device="cuda")
    ws = torch.zeros(H.hkv_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    names = ("k", "v", "pos", "len", "ntok", "nbuf", "qbuf")
    before = {nm: getattr(cb, nm).clone() for nm in names}
    st = torch.cuda.current_stream().cuda_stream
    H.hkv_decode_step(cfg, cb.c, layer, q, k, v, out, ws, ws.numel(), 0, st)
    torch.cuda.synchronize()
    with pytest.raises(H.HkvError) as e:
        H.hkv_check(cb.c)
    assert e.value.status == {"capacity": H.HKV_ERR_CAPACITY, "state": H.HKV_ERR_STATE,
                              "bounds": H.HKV_ERR_BOUNDS}[fault]
    for nm in names:
        assert torch.equal(getattr(cb, nm), before[nm]), nm
    # repaired: the same call takes the step
    field[i] = old
    cb.err.zero_()
    H.hkv_decode_step(cfg, cb.c, layer, q, k, v, out, ws, ws.numel(), 0, st)
    torch.cuda.synchronize()
    H.hkv_check(cb.c)
    ln0 = before["len"].cpu().numpy()
    ln1 = cb.len.cpu().numpy()
    sl = slice(layer * nh, (layer + 1) * nh)
    assert (ln1[sl] == ln0[sl] + 1).all() and (np.delete(ln1, np.r_[sl]) ==
                                                np.delete(ln0, np.r_[sl])).all()
    K = before["k"].float().cpu().numpy()
    Vv = before["v"].float().cpu().numpy()
    off = cb.off.cpu().numpy()
    qn, kn, vn = (x.float().cpu().numpy()[0] for x in (q, k, v))
    got = out.cpu().numpy()[0]
    for h in range(nh):
        o, n_ = int(off[layer * nh + h]), int(ln0[layer * nh + h])
        exp = O.attention(qn[h], np.vstack([K[o:o + n_], kn[h]]), np.vstack([Vv[o:o + n_], vn[h]]))
        assert np.abs(got[h] - exp).max() <= 2e-3, h
