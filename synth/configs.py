"""Workload shapes and hyperparameters for the HeadKV decode path.

These are settings, not arithmetic of the method: both the CPU oracle and
the CUDA path read them and each derives what it needs on its own.

Sources (paper sections / tables):
  * grid and token counts: N = rows x row_len including one end-of-row token
    per row for Lumina-mGPT (Sec. 5.1, Table 3 gives N = 2352 = 48 x 49);
  * recent window w = two grid rows (Sec. 5.1, Implementation Details);
  * grouping trigger E = image tokens generated when head grouping fires:
    100 for Janus-Pro and LlamaGen, 300 for Lumina-mGPT-768, 500 for
    Lumina-mGPT-1024 (Appendix, More Implementation Details);
  * tau = 0.9 (Sec. 4, Step 2) and r_s = 0.5 (Sec. 4, Eq. 5);
  * rho, the fraction of the N image tokens a global head keeps (Sec. 5.1).
The period P of the cache update is not given (Sec. 4, Efficient Cache
Update); it is read here as one grid row. The classification window w_loc is
not given either (Sec. 4, Step 2); it is read as w.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field
from fractions import Fraction

import numpy as np

FP32 = "fp32"
BF16 = "bf16"


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_heads: int
    head_dim: int
    dtype: str
    n_seqs: int
    n_cond: int          # C: conditioning tokens kept by every head
    rows: int            # image grid rows
    row_len: int         # tokens per grid row (incl. end-of-row token)
    recent_w: int        # w
    period: int          # P
    group_at: int        # E (image tokens)
    rho: Fraction        # global-head budget ratio
    tau: float = 0.9
    r_s: float = 0.5
    local_w: int = -1    # w_loc; -1 means "equal to w"
    cfg_rows: int = 1    # sequences per image (2 with classifier-free guidance)
    seed: int = 0
    beta_fixed: tuple | None = None   # per-head beta shared by all layers
    beta_range: tuple = (0.1, 8.0)    # log-uniform range otherwise
    # generator calibration: frequency base of the 2D embedding and query gain
    # kappa (cq = kappa * beta * sqrt(D)); with these, Tiny's beta = 4 heads are
    # local and beta = 0.3 heads global, and on the four model shapes about half
    # of the heads (beta log-uniform in [0.1, 8]) come out local
    pe_base: float = 4.0
    q_gain: float = 6.0

    @property
    def n_image(self) -> int:
        return self.rows * self.row_len

    @property
    def w_loc(self) -> int:
        return self.recent_w if self.local_w < 0 else self.local_w

    @property
    def heads_per_layer(self) -> int:
        return self.n_seqs * self.n_heads

    @property
    def n_head_total(self) -> int:
        return self.n_layers * self.n_seqs * self.n_heads

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == FP32 else 2

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    def beta(self) -> np.ndarray:
        """Per-(layer, head) query scale beta, float64 [L, H]."""
        if self.beta_fixed is not None:
            b = np.asarray(self.beta_fixed, dtype=np.float64)
            assert b.shape == (self.n_heads,)
            return np.tile(b, (self.n_layers, 1))
        rng = np.random.Generator(np.random.PCG64(10_000 + self.seed))
        lo, hi = np.log(self.beta_range[0]), np.log(self.beta_range[1])
        # one draw per (layer, head) of the full model, so that cutting the
        # number of layers keeps the betas of the layers that remain
        return np.exp(rng.uniform(lo, hi, size=(self.n_layers, self.n_heads)))


TINY = Workload(
    name="tiny", n_layers=1, n_heads=8, head_dim=64, dtype=FP32, n_seqs=1,
    n_cond=32, rows=16, row_len=16, recent_w=32, period=16, group_at=32,
    rho=Fraction(1, 4), beta_fixed=(4.0, 4.0, 4.0, 4.0, 0.3, 0.3, 0.3, 0.3),
)

LUMINA_768 = Workload(
    name="lumina768", n_layers=32, n_heads=32, head_dim=128, dtype=BF16,
    n_seqs=16, n_cond=128, rows=48, row_len=49, recent_w=98, period=49,
    group_at=300, rho=Fraction(1, 4),
)

LUMINA_1024 = Workload(
    name="lumina1024", n_layers=32, n_heads=32, head_dim=128, dtype=BF16,
    n_seqs=8, n_cond=128, rows=64, row_len=65, recent_w=130, period=65,
    group_at=500, rho=Fraction(1, 4),
)

LLAMAGEN_XL = Workload(
    name="llamagen_xl", n_layers=36, n_heads=20, head_dim=64, dtype=BF16,
    n_seqs=128, n_cond=1, rows=24, row_len=24, recent_w=48, period=24,
    group_at=100, rho=Fraction(1, 6), cfg_rows=2,
)

JANUS_PRO_7B = Workload(
    name="janus_pro_7b", n_layers=30, n_heads=32, head_dim=128, dtype=BF16,
    n_seqs=64, n_cond=64, rows=24, row_len=24, recent_w=48, period=24,
    group_at=100, rho=Fraction(1, 8), cfg_rows=2,
)

ALL = {w.name: w for w in (TINY, LUMINA_768, LUMINA_1024, LLAMAGEN_XL, JANUS_PRO_7B)}

# rho values swept on the Lumina-mGPT-1024 shape
LUMINA_1024_RHOS = (Fraction(1, 4), Fraction(1, 6), Fraction(1, 8))


def parse_rho(text: str) -> Fraction:
    return Fraction(text)
