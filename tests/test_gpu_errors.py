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
