"""Head-type identification (Sec. 4, Step 2) on the GPU against the oracle
away from the paper's setting: the threshold tau swept over {0.85, 0.95}
(the paper uses 0.9 and reports 0.85-0.95 in its grouping-accuracy study),
and the grouping taken late in the generation instead of at the paper's
early step E; and the multi-query variant (the newest P queries' averaged
attention, each query over the keys of its own step); and the grid-distance
variant (the count runs outward from the current token on the image grid).
Labels must match except declared near-ties; n_h within one."""
import numpy as np
import pytest

from oracle import headkv as O
from synth import configs

from _gpu_util import check_labels, oracle_labels, run_gpu

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,tau", [("lumina768", 0.85), ("lumina768", 0.95),
                                      ("llamagen_xl", 0.85), ("janus_pro_7b", 0.95)])
def test_tau_sweep_labels(name, tau):
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2, tau=tau)
    _, _, labels, nh, _ = run_gpu(w, last_step=w.group_at - 1)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs))
    ties = check_labels(w, labels, nh, lab, f"{name} tau={tau}")
    assert len(ties) <= 2, ties


@pytest.mark.parametrize("name,late", [("llamagen_xl", 400), ("lumina768", 1200)])
def test_late_grouping_labels(name, late):
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2, group_at=late)
    _, _, labels, nh, _ = run_gpu(w, last_step=w.group_at - 1)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs))
    ties = check_labels(w, labels, nh, lab, f"{name} E={late}")
    assert len(ties) <= 2, ties
    g = float((np.asarray(labels) == 1).mean())
    assert 0.0 < g < 1.0, g


@pytest.mark.parametrize("name", ["lumina768", "lumina1024", "llamagen_xl", "janus_pro_7b"])
def test_multi_query_labels(name):
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2)
    _, _, labels, nh, _ = run_gpu(w, last_step=w.group_at - 1, identify="multi")
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs), multi=True)
    ties = check_labels(w, labels, nh, lab, f"{name} multi")
    assert len(ties) <= 2, ties
    # every margin is far from tau here, so n_h was compared for every head
    assert min(m for res in lab.values() for (_, _, m, _) in res) > 1e-3


@pytest.mark.parametrize("name", ["llamagen_xl", "lumina768"])
def test_multi_query_labels_grouping_at_the_period(name):
    """E = P: every image token's query counts, the oldest over only the
    conditioning tokens and itself."""
    w0 = configs.ALL[name]
    w = w0.with_(n_layers=1, n_seqs=2, group_at=w0.period)
    _, _, labels, nh, _ = run_gpu(w, last_step=w.group_at - 1, identify="multi")
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs), multi=True)
    ties = check_labels(w, labels, nh, lab, f"{name} E=P multi")
    assert len(ties) <= 2, ties


@pytest.mark.parametrize("name", ["lumina768", "lumina1024", "llamagen_xl", "janus_pro_7b"])
def test_grid_distance_labels(name):
    w = configs.ALL[name].with_(n_layers=2, n_seqs=2)
    _, _, labels, nh, _ = run_gpu(w, last_step=w.group_at - 1, distance_mode=O.GRID2D)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs), distance=O.GRID2D)
    ties = check_labels(w, labels, nh, lab, f"{name} grid")
    assert len(ties) <= 2, ties


def test_grid_distance_multi_query_labels():
    # the queries' own neighbourhoods lie away from the current token on the
    # grid, so the averaged count is long: every head comes out global here
    w = configs.ALL["janus_pro_7b"].with_(n_layers=2, n_seqs=2)
    _, _, labels, nh, _ = run_gpu(w, last_step=w.group_at - 1, identify="multi",
                                  distance_mode=O.GRID2D)
    lab = oracle_labels(w, range(w.n_layers), range(w.n_seqs), multi=True, distance=O.GRID2D)
    ties = check_labels(w, labels, nh, lab, "janus grid multi")
    assert not ties
