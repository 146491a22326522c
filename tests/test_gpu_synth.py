"""The GPU twin of the input generator writes the same bits as synth/gen.py."""
import numpy as np
import pytest

from synth import configs, gen

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", list(configs.ALL))
def test_device_generator_is_bit_identical(name):
    torch = pytest.importorskip("torch")
    from synth.gpu import DeviceSynth
    w0 = configs.ALL[name]
    w = w0.with_(n_layers=min(w0.n_layers, 3), n_seqs=min(w0.n_seqs, 3))
    dt = torch.bfloat16 if w.dtype == configs.BF16 else torch.float32
    ds = DeviceSynth(w, "cuda")
    S, H, D = w.n_seqs, w.n_heads, w.head_dim
    nl, nt, t0 = w.n_layers, 3, w.n_image - 3
    q = torch.empty(nt, nl, S, H, D, dtype=dt, device="cuda")
    k, v = torch.empty_like(q), torch.empty_like(q)
    ds.image(q, k, v, 0, nl, t0, nt)
    pe, cq = gen.pe_table(w), gen.q_coef(w)
    for tt in range(nt):
        for l in range(nl):
            rq, rk, rv = gen.layer_step(w, l, t0 + tt, pe, cq)
            for got, ref in ((q, rq), (k, rk), (v, rv)):
                g = got[tt, l].float().cpu().numpy()
                assert np.array_equal(g.view(np.uint32), ref.view(np.uint32))
    ds.image(q[:1], k[:1], v[:1], 0, nl, 0, 1)
    for l in range(nl):
        rq, rk, rv = gen.layer_step(w, l, 0, pe, cq)
        assert np.array_equal(q[0, l].float().cpu().numpy().view(np.uint32), rq.view(np.uint32))
    if w.n_cond:
        kc = torch.empty(S, H, w.n_cond, D, dtype=dt, device="cuda")
        vc = torch.empty_like(kc)
        ds.cond(kc, vc, 1)
        rk, rv = gen.layer_cond(w, 1)
        assert np.array_equal(kc.float().cpu().numpy().view(np.uint32), rk.view(np.uint32))
        assert np.array_equal(vc.float().cpu().numpy().view(np.uint32), rv.view(np.uint32))
