"""The C-ABI library without a GPU: it loads, exports every entry point the
header declares, and its host-side validation and fault injection answer
before any CUDA call."""
import ctypes
import os
import re

import pytest

from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "hkv.h")


@pytest.fixture(scope="module")
def H():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2605_20600_gb300 import hkv
    hkv.lib()
    return hkv


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hkv_[a-z_]+)\s*\(", text)))


def tiny_cfg(H, **kw):
    base = dict(n_layers=2, n_seqs=2, n_heads=4, head_dim=64, dtype="bf16", n_cond=8, n_image=64,
                row_len=8, recent_w=16, local_w=16, period=8, group_at=16, global_budget=24)
    base.update(kw)
    return H.make_config(**base)


def fake_cache(H, **kw):
    # aligned, non-null host addresses: never dereferenced by the checks tested here
    buf = ctypes.create_string_buffer(4096)
    a = (ctypes.addressof(buf) + 255) & ~255
    c = H.hkv_cache(a, a + 256, a, a, a, a, a, a, a, a + 512, a, 1000)
    for k, v in kw.items():
        setattr(c, k, v)
    c._keep = buf
    return c


def test_every_declared_symbol_is_exported(H):
    names = declared_functions()
    assert len(names) == 21
    for n in names:
        assert hasattr(H.lib(), n), n
    assert set(names) >= {"hkv_identify_heads", "hkv_allocate_budgets", "hkv_append_evict",
                          "hkv_decode_attention"}


def test_struct_sizes(H):
    assert ctypes.sizeof(H.hkv_config) == 16 * 4 + 2 * 8
    assert ctypes.sizeof(H.hkv_cache) == 11 * 8 + 8


def test_status_strings(H):
    assert H.hkv_status_str(0) == "ok"
    assert "capacity" in H.hkv_status_str(3)
    assert H.hkv_status_str(99) == "unknown status"


@pytest.mark.parametrize("change,code", [
    (dict(head_dim=96), 2), (dict(dtype=5), 1), (dict(period=32), 2), (dict(global_budget=8), 2),
    (dict(global_budget=65), 2), (dict(group_at=65), 2), (dict(n_seqs=0), 2), (dict(tau=0.0), 1),
    (dict(r_s=1.5), 1), (dict(budget_mode=2), 1), (dict(distance_mode=2), 1), (dict(reserved=1), 1),
    # squared grid distances of a 50000 x 1 grid do not fit 31 bits
    (dict(distance_mode=1, row_len=1, n_image=50000), 2),
])
def test_validate_config_rejects(H, change, code):
    cfg = tiny_cfg(H)
    for k, v in change.items():
        setattr(cfg, k, v)
    with pytest.raises(H.HkvError) as e:
        H.hkv_validate_config(cfg)
    assert e.value.status == code


def test_validate_config_accepts_paper_shapes(H):
    from fractions import Fraction
    from synth import configs
    for w in configs.ALL.values():
        cfg = H.make_config(n_layers=w.n_layers, n_seqs=w.n_seqs, n_heads=w.n_heads,
                            head_dim=w.head_dim, dtype=w.dtype, n_cond=w.n_cond,
                            n_image=w.n_image, row_len=w.row_len, recent_w=w.recent_w,
                            local_w=w.w_loc, period=w.period, group_at=w.group_at, rho=w.rho)
        H.hkv_validate_config(cfg)
        assert H.hkv_workspace_size(cfg) > 0
    assert H.make_config(**{**dict(n_layers=1, n_seqs=1, n_heads=1, head_dim=128, dtype="bf16",
                                   n_cond=128, n_image=4160, row_len=65, recent_w=130,
                                   local_w=130, period=65, group_at=500)},
                         rho=Fraction(1, 6)).global_budget == 693


def test_workspace_size_zero_for_bad_config(H):
    assert H.hkv_workspace_size(tiny_cfg(H, head_dim=32)) == 0


def test_null_and_misaligned_arguments(H):
    cfg = tiny_cfg(H)
    c = fake_cache(H)
    lib = H.lib()
    assert lib.hkv_decode_attention(ctypes.byref(cfg), None, 0, 16, 16, 16, 1 << 30, None) == 1
    assert lib.hkv_decode_attention(ctypes.byref(cfg), ctypes.byref(c), 0, None, 16, 16, 1 << 30, None) == 1
    assert lib.hkv_decode_attention(ctypes.byref(cfg), ctypes.byref(c), 0, 24, 16, 16, 1 << 30, None) == 8
    assert lib.hkv_decode_attention(ctypes.byref(cfg), ctypes.byref(c), 2, 16, 16, 16, 1 << 30, None) == 1
    assert lib.hkv_decode_attention(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 8, None) == 3
    assert lib.hkv_append_evict(ctypes.byref(cfg), ctypes.byref(c), -1, 16, 16, 16, None) == 1
    assert lib.hkv_append_evict(ctypes.byref(cfg), ctypes.byref(c), 0, 16, None, 16, None) == 1
    bad = fake_cache(H, qbuf=c.qbuf + 8)
    assert lib.hkv_append_evict(ctypes.byref(cfg), ctypes.byref(bad), 0, 16, 16, 16, None) == 8
    nul = fake_cache(H, err=None)
    assert lib.hkv_identify_heads(ctypes.byref(cfg), ctypes.byref(nul), 0, 16, 16, None, None) == 1
    assert lib.hkv_identify_heads_multi(ctypes.byref(cfg), ctypes.byref(nul), 0, 16, None, None) == 1
    assert lib.hkv_identify_heads_multi(ctypes.byref(cfg), ctypes.byref(c), 0, None, None, None) == 1
    assert lib.hkv_identify_heads_multi(ctypes.byref(cfg), ctypes.byref(c), 2, 16, None, None) == 1
    small = fake_cache(H, capacity_tokens=10)
    assert lib.hkv_init_dense(ctypes.byref(cfg), ctypes.byref(small), None) == 3
    other = fake_cache(H, qbuf=c.qbuf + 256)
    assert lib.hkv_repack(ctypes.byref(cfg), ctypes.byref(c), ctypes.byref(other), 0, None) == 1
    assert lib.hkv_allocate_budgets(ctypes.byref(cfg), None, 16, 16, 16, None, None) == 1
    assert lib.hkv_check(None, None) == 1
    assert lib.hkv_decode_step(ctypes.byref(cfg), ctypes.byref(c), 0, 16, None, 16, 16, 16, 1 << 30, 0, None) == 1
    assert lib.hkv_decode_step(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 16, 16, 8, 0, None) == 3
    assert lib.hkv_decode_step(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 24, 16, 16, 16, 1 << 30, 0, None) == 8
    assert lib.hkv_decode_step(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 16, 16, 1 << 30, 6, None) == 1
    assert lib.hkv_evict(ctypes.byref(cfg), ctypes.byref(c), 5, None) == 1
    assert lib.hkv_evict_all(ctypes.byref(cfg), None, None) == 1
    assert lib.hkv_evict_all(None, ctypes.byref(c), None) == 1
    assert lib.hkv_evict_all(ctypes.byref(tiny_cfg(H, head_dim=32)), ctypes.byref(c), None) == 2
    cnt = ctypes.c_int64(0)
    assert lib.hkv_export_state(ctypes.byref(cfg), None, 0, None, None, None, None, None, 0,
                                ctypes.byref(cnt), None) == 1
    assert lib.hkv_export_state(ctypes.byref(cfg), ctypes.byref(c), 2, None, None, None, None, None,
                                0, ctypes.byref(cnt), None) == 1
    assert lib.hkv_export_state(ctypes.byref(cfg), ctypes.byref(c), 0, None, None, None, None, 16,
                                -1, ctypes.byref(cnt), None) == 1
    assert lib.hkv_decode_step_identify(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 16, None,
                                        16, 1 << 30, 0, None) == 1
    assert lib.hkv_decode_step_identify(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 16, 16,
                                        16, 8, 0, None) == 3
    grid = tiny_cfg(H)
    grid.distance_mode = 1
    H.hkv_validate_config(grid)
    assert lib.hkv_decode_step_identify(ctypes.byref(grid), ctypes.byref(c), 0, 16, 16, 16, 16, 16,
                                        16, 1 << 30, 0, None) == 1
    nopos = fake_cache(H, pos=None)
    assert lib.hkv_export_state(ctypes.byref(cfg), ctypes.byref(nopos), 0, None, None, None, None,
                                16, 8, ctypes.byref(cnt), None) == 1


@pytest.mark.parametrize("name", ["decode_attention", "append_evict", "identify_heads",
                                  "allocate_budgets", "repack", "prefill", "init_dense", "check",
                                  "decode_step", "evict", "evict_all", "export_state",
                                  "decode_step_identify", "identify_heads_multi"])
def test_fault_injection_returns_the_code(H, name, monkeypatch):
    cfg = tiny_cfg(H)
    c = fake_cache(H)
    monkeypatch.setenv("HKV_FAULT_INJECT", f"{name}:6")
    lib = H.lib()
    calls = {
        "decode_attention": lambda: lib.hkv_decode_attention(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 1 << 30, None),
        "append_evict": lambda: lib.hkv_append_evict(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, None),
        "identify_heads": lambda: lib.hkv_identify_heads(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, None, None),
        "identify_heads_multi": lambda: lib.hkv_identify_heads_multi(ctypes.byref(cfg), ctypes.byref(c), 0, 16, None, None),
        "allocate_budgets": lambda: lib.hkv_allocate_budgets(ctypes.byref(cfg), 16, 16, 16, 16, None, None),
        "repack": lambda: lib.hkv_repack(ctypes.byref(cfg), ctypes.byref(c), ctypes.byref(c), 0, None),
        "prefill": lambda: lib.hkv_prefill(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, None),
        "init_dense": lambda: lib.hkv_init_dense(ctypes.byref(cfg), ctypes.byref(c), None),
        "check": lambda: lib.hkv_check(ctypes.byref(c), None),
        "decode_step": lambda: lib.hkv_decode_step(ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 16, 16, 1 << 30, 0, None),
        "evict": lambda: lib.hkv_evict(ctypes.byref(cfg), ctypes.byref(c), 0, None),
        "evict_all": lambda: lib.hkv_evict_all(ctypes.byref(cfg), ctypes.byref(c), None),
        "decode_step_identify": lambda: lib.hkv_decode_step_identify(
            ctypes.byref(cfg), ctypes.byref(c), 0, 16, 16, 16, 16, 16, 16, 1 << 30, 0, None),
        "export_state": lambda: lib.hkv_export_state(ctypes.byref(cfg), ctypes.byref(c), 0, None, None,
                                                     None, None, None, 0, None, None),
    }
    assert calls[name]() == 6


def test_fault_injection_raises_through_binding(H, monkeypatch):
    c = fake_cache(H)
    monkeypatch.setenv("HKV_FAULT_INJECT", "check:6")
    with pytest.raises(H.HkvError) as e:
        H.hkv_check(c)
    assert e.value.status == 6 and "timed out" in str(e.value)


def test_fault_injection_other_name_does_not_fire(H, monkeypatch):
    monkeypatch.setenv("HKV_FAULT_INJECT", "repack:6")
    H.hkv_validate_config(tiny_cfg(H))


@pytest.mark.parametrize("fused,identify,distance,ok", [
    (True, "fused", 0, True), (True, "separate", 1, True), (True, "multi", 1, True),
    (False, "fused", 0, False), (True, "fused", 1, False), (True, "bogus", 0, False),
    # the default: fused where the distances are raster, separate otherwise
    (True, None, 0, True), (True, None, 1, True), (False, None, 1, True)])
def test_runner_identification_choices(H, fused, identify, distance, ok):
    """The runner refuses combinations the library cannot run before it
    touches the device (a stand-in engine with a configuration only)."""
    from paper_2605_20600_gb300.runner import generate

    class Stop(Exception):
        pass

    class FakeEngine:
        cfg = tiny_cfg(H, distance_mode=distance)

        @property
        def device(self):
            raise Stop()   # the first device access: the checks have passed

    with pytest.raises(Stop if ok else ValueError):
        generate(FakeEngine(), None, fused=fused, identify=identify)



def test_missing_library_fails_loudly(H, monkeypatch, tmp_path):
    """No CPU fallback: without libheadkv.so every call raises."""
    monkeypatch.setattr(H, "_lib", None)
    monkeypatch.setattr(H, "LIB_PATH", str(tmp_path / "libheadkv.so"))
    with pytest.raises(RuntimeError, match="missing"):
        H.hkv_validate_config(tiny_cfg(H))
    with pytest.raises(RuntimeError, match="missing"):
        H.hkv_check(fake_cache(H))


@pytest.mark.parametrize("period,group_at", [(16, 32), (1, 20), (5, 5), (7, 40)])
def test_engine_update_schedule_matches_the_oracle(H, period, group_at):
    """The steps at which the engine runs the periodic update (R7) are the
    steps at which the oracle's generation does."""
    from oracle import headkv as O
    from synth import configs, gen
    from paper_2605_20600_gb300.engine import Engine
    w = configs.TINY.with_(period=period, group_at=group_at)
    hi = gen.HeadInputs(w, 0, 0, 5)
    tr = O.run_head(O.HeadParams.of(w), hi.q, hi.k, hi.v)
    oracle_steps = [u.t_last + 1 for u in tr.updates[1:]]     # [0] is the grouping update

    class Cfg:
        pass
    fake = Cfg()
    fake.cfg = tiny_cfg(H, period=period, group_at=group_at, n_image=w.n_image)
    assert [t for t in range(w.n_image) if Engine.update_due(fake, t)] == oracle_steps


def test_global_budget_is_the_oracle_rule(H):
    """hkv_global_budget (Sec. 5.1, B_g = floor(rho N)) against the oracle's
    global_budget: Table 3's B column and a sweep of ratios and grid sizes."""
    from fractions import Fraction
    from oracle import headkv as O
    assert H.hkv_global_budget(Fraction(1, 4), 576) == 144
    assert H.hkv_global_budget(Fraction(1, 6), 576) == 96
    assert H.hkv_global_budget(Fraction(1, 8), 576) == 72
    assert H.hkv_global_budget(Fraction(1, 8), 2352) == 294
    for den in range(1, 13):
        for num in range(1, den + 1):
            for n in (1, 7, 256, 576, 2352, 4160, 9999):
                r = Fraction(num, den)
                assert H.hkv_global_budget(r, n) == O.global_budget(r, n), (r, n)
    lib = H.lib()
    out = ctypes.c_int32(0)
    for args in [(0, 4, 100), (5, 4, 100), (1, 0, 100), (1, 4, 0), (-1, 4, 100), (1, 1 << 40, 10)]:
        assert lib.hkv_global_budget(*args, ctypes.byref(out)) == 1, args
    assert lib.hkv_global_budget(1, 4, 100, None) == 1


def test_update_due_rejects_bad_arguments(H):
    lib = H.lib()
    out = ctypes.c_int32(0)
    cfg = tiny_cfg(H)
    assert lib.hkv_update_due(ctypes.byref(cfg), -1, ctypes.byref(out)) == 1
    assert lib.hkv_update_due(ctypes.byref(cfg), 3, None) == 1
    assert lib.hkv_update_due(ctypes.byref(tiny_cfg(H, head_dim=32)), 3, ctypes.byref(out)) == 2


def test_decode_step_launches_answers_zero_for_a_bad_config(H):
    assert H.lib().hkv_decode_step_launches(ctypes.byref(tiny_cfg(H, head_dim=32))) == 0


def test_noalloc_host_checks_answer_before_the_device(H, monkeypatch):
    """hkv_decode_attention_noalloc validates its arguments on the host (no
    CUDA call: this runs without a GPU) and honours fault injection."""
    f = H.lib().hkv_decode_attention_noalloc
    f.argtypes = [ctypes.POINTER(H.hkv_config), ctypes.POINTER(H.hkv_cache), ctypes.c_int,
                  ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int
    cfg = tiny_cfg(H)
    c = fake_cache(H)
    q = out = c.k  # aligned, never dereferenced by the checks
    assert f(ctypes.byref(tiny_cfg(H, head_dim=32)), ctypes.byref(c), 0, q, out, None) == 2
    assert f(ctypes.byref(cfg), None, 0, q, out, None) == 1
    for field in ("k", "v", "off", "len", "err"):
        assert f(ctypes.byref(cfg), ctypes.byref(fake_cache(H, **{field: None})), 0, q, out,
                 None) == 1, field
    assert f(ctypes.byref(cfg), ctypes.byref(c), 0, None, out, None) == 1
    assert f(ctypes.byref(cfg), ctypes.byref(c), 0, q, None, None) == 1
    assert f(ctypes.byref(cfg), ctypes.byref(c), 0, q + 8, out, None) == 8
    assert f(ctypes.byref(cfg), ctypes.byref(c), 0, q, out + 4, None) == 8
    assert f(ctypes.byref(cfg), ctypes.byref(fake_cache(H, k=c.k + 8)), 0, q, out, None) == 8
    assert f(ctypes.byref(cfg), ctypes.byref(c), 2, q, out, None) == 1   # n_layers = 2
    assert f(ctypes.byref(cfg), ctypes.byref(c), -1, q, out, None) == 1
    monkeypatch.setenv("HKV_FAULT_INJECT", "decode_attention_noalloc:6")
    assert f(ctypes.byref(cfg), ctypes.byref(c), 0, q, out, None) == 6
