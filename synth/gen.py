"""Seeded, counter-based synthetic Q/K/V shaped like an AR image model.

This module is the definition of the inputs. It holds no arithmetic of the
HeadKV method. The CPU oracle and the CUDA path both consume its values; the
GPU twin of this generator (synth_gpu.cu) reproduces these exact bits, and a
GPU test checks that.

Definition (every step is exact or a single IEEE-754 round-to-nearest op, so
that two implementations agree bit for bit):

  * u = SplitMix64(seed) output number n, i.e. z = seed + (n+1)*0x9E3779B97F4A7C15
    (mod 2^64) followed by SplitMix64's published finaliser
    (xor-shift 30, *0xBF58476D1CE4E5B9, xor-shift 27, *0x94D049BB133111EB,
    xor-shift 31).
  * n = ((((((tensor*1024 + s)*128 + l)*128 + h)*16384 + tok)*256) + d)
    with tensor 0/1/2 for q/k/v, s the sequence, l the layer, h the head,
    tok the token index in the cache (conditioning tokens 0..C-1, image token
    t at C+t) and d the channel.
  * g = (sum of the four 16-bit fields of u) - 131070, an integer whose
    distribution (Irwin-Hall of 4) approximates N(0, var) with
    var = (65536^2 - 1)/3; it is exact in fp32.
  * noise = fp32(g) * S where S is a float32 constant: KS = fp32(0.1/std)
    for q and k, VS = fp32(1/std) for v.
  * pe[r][c] is a 2D sinusoidal embedding of the grid position (row r,
    column c) of an image token, computed in fp64 and rounded to fp32 once;
    D/2 channels encode r and D/2 encode c, each half of unit norm.
  * image token t at (r, c) = divmod(t, row_len):
        k = pe[r][c] + noise_k
        q = cq[l][h] * pe[r][c] + noise_q,   cq = fp32(kappa * beta[l][h] * sqrt(D))
        v = noise_v
    conditioning tokens: k = noise_k, v = noise_v (they have no grid position).
  * the fp32 value is rounded to the workload dtype (bf16: round to nearest
    even on the top 16 bits).

So q.k / sqrt(D) ~ kappa * beta * pe.pe', i.e. beta sets how sharply a head's
attention falls off with 2D distance on the grid: large beta gives a
locality-biased head, small beta a broad one.
"""
from __future__ import annotations

import numpy as np

from .configs import BF16, FP32, Workload

TENSOR_Q, TENSOR_K, TENSOR_V = 0, 1, 2

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_MASK16 = np.uint64(0xFFFF)

IH_STD = float(np.sqrt((65536.0 ** 2 - 1.0) / 3.0))
KS = np.float32(0.1 / IH_STD)
VS = np.float32(1.0 / IH_STD)

MAX_SEQS, MAX_LAYERS, MAX_HEADS, MAX_TOKENS, MAX_DIM = 1024, 128, 128, 16384, 256


def splitmix64(seed: int, n) -> np.ndarray:
    """Output number n (n >= 0) of SplitMix64 seeded with `seed`, as uint64."""
    n = np.asarray(n, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (n + np.uint64(1)) * _GAMMA
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def counter(tensor, s, l, h, tok, d) -> np.ndarray:
    c = np.uint64(tensor)
    for x, width in ((s, 1024), (l, 128), (h, 128), (tok, 16384), (d, 256)):
        c = c * np.uint64(width) + np.asarray(x, dtype=np.uint64)
    return c


def irwin_hall4(u: np.ndarray) -> np.ndarray:
    a = (u & _MASK16) + ((u >> np.uint64(16)) & _MASK16) \
        + ((u >> np.uint64(32)) & _MASK16) + ((u >> np.uint64(48)) & _MASK16)
    return a.astype(np.int64) - 131070


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even); float32 out."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    with np.errstate(over="ignore"):
        r = (u + rounding) & np.uint32(0xFFFF0000)
    return r.view(np.float32)


def to_dtype(x: np.ndarray, dtype: str) -> np.ndarray:
    return round_bf16(x) if dtype == BF16 else np.asarray(x, dtype=np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Top 16 bits of float32 values that are already bf16-representable."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def pe_table(w: Workload) -> np.ndarray:
    """2D sinusoidal embedding, float32 [rows, row_len, D]."""
    D = w.head_dim
    half = D // 2
    nf = half // 2
    omega = w.pe_base ** (-np.arange(nf, dtype=np.float64) / nf)

    def axis(n):
        ang = np.arange(n, dtype=np.float64)[:, None] * omega[None, :]
        e = np.empty((n, half), dtype=np.float64)
        e[:, 0::2] = np.sin(ang)
        e[:, 1::2] = np.cos(ang)
        return e / np.sqrt(nf)

    er, ec = axis(w.rows), axis(w.row_len)
    pe = np.empty((w.rows, w.row_len, D), dtype=np.float64)
    pe[:, :, :half] = er[:, None, :]
    pe[:, :, half:] = ec[None, :, :]
    return pe.astype(np.float32)


def q_coef(w: Workload) -> np.ndarray:
    """cq = fp32(kappa * beta * sqrt(D)), float32 [L, H]."""
    return (w.q_gain * w.beta() * np.sqrt(float(w.head_dim))).astype(np.float32)


def _check(w: Workload):
    assert w.n_seqs <= MAX_SEQS and w.n_layers <= MAX_LAYERS and w.n_heads <= MAX_HEADS
    assert w.n_cond + w.n_image <= MAX_TOKENS and w.head_dim <= MAX_DIM


def _noise(w: Workload, tensor, s, l, h, tok) -> np.ndarray:
    """fp32(g) for tokens `tok` (1-D) of one head: float32 [len(tok), D]."""
    d = np.arange(w.head_dim, dtype=np.uint64)[None, :]
    tok = np.asarray(tok, dtype=np.uint64)[:, None]
    g = irwin_hall4(splitmix64(w.seed, counter(tensor, s, l, h, tok, d)))
    return g.astype(np.float32)


class HeadInputs:
    """Inputs of one head (s, l, h) of a workload.

    q[t] is the query of image token t (t in 0..N-1); k[j], v[j] are the key
    and value of cache token j (j < C conditioning, j = C+t image token t).
    Values are float32 arrays holding dtype-exact numbers.
    """

    def __init__(self, w: Workload, s: int, l: int, h: int, pe=None, cq=None):
        _check(w)
        self.w, self.s, self.l, self.h = w, s, l, h
        pe = pe_table(w) if pe is None else pe
        cq = q_coef(w) if cq is None else cq
        C, N, D = w.n_cond, w.n_image, w.head_dim
        t = np.arange(N)
        pe_t = pe[t // w.row_len, t % w.row_len, :]                 # [N, D]
        nq = _noise(w, TENSOR_Q, s, l, h, C + t)
        self.q = to_dtype(cq[l, h] * pe_t + nq * KS, w.dtype)
        j = np.arange(C + N)
        nk = _noise(w, TENSOR_K, s, l, h, j) * KS
        k = nk.copy()
        k[C:] = pe_t + nk[C:]
        self.k = to_dtype(k, w.dtype)
        self.v = to_dtype(_noise(w, TENSOR_V, s, l, h, j) * VS, w.dtype)


def layer_step(w: Workload, l: int, t: int, pe=None, cq=None):
    """q, k, v of image token t for every (s, h) of layer l: float32 [S, H, D]."""
    _check(w)
    pe = pe_table(w) if pe is None else pe
    cq = q_coef(w) if cq is None else cq
    S, H, D, C = w.n_seqs, w.n_heads, w.head_dim, w.n_cond
    s = np.arange(S, dtype=np.uint64)[:, None, None]
    h = np.arange(H, dtype=np.uint64)[None, :, None]
    d = np.arange(D, dtype=np.uint64)[None, None, :]
    tok = np.uint64(C + t)

    def noise(tensor):
        return irwin_hall4(splitmix64(w.seed, counter(tensor, s, l, h, tok, d))).astype(np.float32)

    pe_t = pe[t // w.row_len, t % w.row_len, :][None, None, :]
    q = to_dtype(cq[l][None, :, None] * pe_t + noise(TENSOR_Q) * KS, w.dtype)
    k = to_dtype(pe_t + noise(TENSOR_K) * KS, w.dtype)
    v = to_dtype(noise(TENSOR_V) * VS, w.dtype)
    return q, k, v


def layer_cond(w: Workload, l: int):
    """k, v of the C conditioning tokens of layer l: float32 [S, H, C, D]."""
    _check(w)
    S, H, D, C = w.n_seqs, w.n_heads, w.head_dim, w.n_cond
    s = np.arange(S, dtype=np.uint64)[:, None, None, None]
    h = np.arange(H, dtype=np.uint64)[None, :, None, None]
    j = np.arange(C, dtype=np.uint64)[None, None, :, None]
    d = np.arange(D, dtype=np.uint64)[None, None, None, :]

    def noise(tensor):
        return irwin_hall4(splitmix64(w.seed, counter(tensor, s, l, h, j, d))).astype(np.float32)

    return to_dtype(noise(TENSOR_K) * KS, w.dtype), to_dtype(noise(TENSOR_V) * VS, w.dtype)
