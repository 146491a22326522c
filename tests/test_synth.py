"""The shared input generator: SplitMix64 against its published outputs,
bf16 rounding, determinism and the noise moments."""
import numpy as np
import pytest

from synth import configs, gen


def test_splitmix64_published_sequence():
    # first outputs of SplitMix64 seeded with 0 (Steele, Lea & Flood 2014;
    # the reference C implementation by S. Vigna)
    got = gen.splitmix64(0, np.arange(3))
    assert [int(x) for x in got] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_bf16_round_nearest_even():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(size=10000).astype(np.float32) * 10,
                        np.float32([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8, 0.0, -0.0])])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(gen.round_bf16(x).view(np.uint32), ref.view(np.uint32))
    assert gen.round_bf16(np.float32([1.0 + 2 ** -8]))[0] == 1.0          # tie -> even
    assert gen.round_bf16(np.float32([1.0 + 3 * 2 ** -8]))[0] == 1.0 + 2 ** -6


def test_head_inputs_agree_with_layer_slices():
    w = configs.LLAMAGEN_XL.with_(n_layers=2, n_seqs=3)
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    hi = gen.HeadInputs(w, 2, 1, 7, pe, cq)
    for t in (0, 5, 575):
        q, k, v = gen.layer_step(w, 1, t, pe, cq)
        assert np.array_equal(q[2, 7], hi.q[t])
        assert np.array_equal(k[2, 7], hi.k[w.n_cond + t])
        assert np.array_equal(v[2, 7], hi.v[w.n_cond + t])
    kc, vc = gen.layer_cond(w, 1)
    assert np.array_equal(kc[2, 7], hi.k[: w.n_cond]) and np.array_equal(vc[2, 7], hi.v[: w.n_cond])


def test_deterministic_and_seed_dependent():
    w = configs.TINY
    a = gen.HeadInputs(w, 0, 0, 3)
    b = gen.HeadInputs(w, 0, 0, 3)
    c = gen.HeadInputs(w.with_(seed=1), 0, 0, 3)
    assert np.array_equal(a.k, b.k) and not np.array_equal(a.v, c.v)


def test_values_are_dtype_exact():
    w = configs.JANUS_PRO_7B.with_(n_layers=1)
    hi = gen.HeadInputs(w, 0, 0, 0)
    for x in (hi.q, hi.k, hi.v):
        assert np.array_equal(gen.round_bf16(x), x)


def test_noise_moments():
    w = configs.LUMINA_1024.with_(n_layers=1)
    v = gen.HeadInputs(w, 0, 0, 0).v
    assert abs(v.mean()) < 0.01 and abs(v.std() - 1.0) < 0.01
    assert np.abs(v).max() <= np.sqrt(3.0) * 2 + 1e-3      # Irwin-Hall(4) support


def test_pe_halves_have_unit_norm():
    w = configs.LUMINA_768
    pe = gen.pe_table(w).astype(np.float64)
    half = w.head_dim // 2
    np.testing.assert_allclose((pe[..., :half] ** 2).sum(-1), 1.0, atol=1e-6)
    np.testing.assert_allclose((pe[..., half:] ** 2).sum(-1), 1.0, atol=1e-6)
