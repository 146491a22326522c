"""CPU oracle of the HeadKV decode path.

TEST INFRASTRUCTURE ONLY: tests/, __graft_entry__.smoke() and the CPU
baseline leg of bench.py may import this module; the product path never
does. It shares no code with the CUDA path.

Each function follows one passage of the paper "Head-Aware Key-Value
Compression for Efficient Autoregressive Image Generation" (HeadKV):

  attention          Eq. 1 (Sec. 3), fp64 brute force
  grouping_count     Sec. 4 Step 2 (threshold-based attention accumulation)
  classify           Sec. 4 Step 2 (local iff the count is below w_loc)
  grouping_count_multi  a variant of Step 2 not in the paper: the buffered
                     queries' attention averaged, each over its own prefix
  grid_d2, count_order_2d, grouping_count_2d, grouping_count_multi_2d
                     a variant of Step 2 not in the paper: the count runs
                     outward from the current token by distance on the image
                     grid instead of backward in raster order
  global_budget      Sec. 5.1 Implementation Details (rho * N tokens)
  redistributed_budgets  a budget variant not in the paper: local heads'
                     unused tokens shared among the group's global heads
  arena_layout       Sec. 5.1 (local heads keep w, global heads rho*N) and
                     Sec. 4 Efficient Cache Update (room for P buffered tokens)
  ste_partition      Eq. 5 (long/near split by r_s)
  ste_long_2d, ste_evict_strata
                     a variant of Eq. 5 not in the paper: the long-range
                     subset is the T r_s history tokens farthest on the grid
  ste_scores_eq6     Eq. 6 as printed, fp64
  ste_scores_fp32    Eq. 6 ranking in the precision the decision is taken in
  ste_quotas         Sec. 4 STE (M/2 evicted from each subset)
  ste_evict          Sec. 4 STE (lowest scores evicted, survivors concatenated)
  cache_update       Eqs. 2-4 (cache = [cond, history, recent]; local heads
                     drop history, global heads apply STE to it)
  run_head           Steps 1-3 with the periodic update, one head end to end

Readings where the paper is silent (each is listed with its reason in the
design notes of the repository):
  * E counts image tokens; grouping uses the query of image token E-1 over
    the dense cache after that token is appended, once per (seq, layer, head).
  * the backward count includes the current token and may run into the
    conditioning tokens; local iff n_h < w_loc, w_loc = w.
  * global heads keep B_g = floor(rho*N) image tokens (history + recent) plus
    the C conditioning tokens; local heads keep w image tokens plus C.
  * P new tokens are buffered; when the buffer is full the update runs after
    that step's attention (i.e. at the start of the next step); the grouping
    step's update runs after the attention of image token E-1.
  * Q_past = the queries of the P most recently appended image tokens.
  * Eq. 5 splits the T history tokens at n_long = floor(T * r_s) (fp64);
    M_long = floor(M/2), M_near = M - M_long; a stratum with fewer tokens
    than its quota passes the excess to the other.
  * ties in score evict the older token (smaller position) first.
  * the ranking decision is taken in fp32 with a fixed operation order
    (ste_scores_fp32); ste_scores_eq6 is the literal fp64 formula, used to
    check that the fp32 decision ranks like Eq. 6 away from near-ties.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from fractions import Fraction

import numpy as np

LOCAL, GLOBAL = 0, 1


# ----------------------------------------------------------------------------
# Eq. 1: O = Softmax(Q K^T / sqrt(d)) V, one query row
# ----------------------------------------------------------------------------
def attention(q, K, V) -> np.ndarray:
    """softmax(q K^T / sqrt(d)) V for a single query q [d], K, V [n, d]; fp64."""
    q = np.asarray(q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    if K.shape[0] == 0:
        return np.zeros(V.shape[1], dtype=np.float64)
    logits = (K @ q) / math.sqrt(q.shape[0])
    p = np.exp(logits - logits.max())
    return (p @ V) / p.sum()


def attention_weights(q, K) -> np.ndarray:
    q = np.asarray(q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    logits = (K @ q) / math.sqrt(q.shape[0])
    p = np.exp(logits - logits.max())
    return p / p.sum()


# ----------------------------------------------------------------------------
# Sec. 4 Step 2: head grouping
# ----------------------------------------------------------------------------
def grouping_count(q, K, tau: float):
    """Attention of the current query over the key cache K (oldest first),
    accumulated backward from the current (newest) position until tau is
    reached. Returns (n_h, cum) with cum[n-1] = mass of the newest n tokens
    and n_h the minimum n with cum[n-1] >= tau."""
    p = attention_weights(q, K)
    cum = np.cumsum(p[::-1])
    hit = np.nonzero(cum >= tau)[0]
    n_h = int(hit[0]) + 1 if hit.size else int(cum.size)
    return n_h, cum


def grouping_count_multi(Q, K, tau: float):
    """Multi-query variant of Step 2 (not in the paper): the P buffered
    queries Q [P, d] (oldest first, the last is the current token's) each
    attend over the cache as it stood at their own step (query p of P sees
    the oldest len(K) - (P - 1 - p) keys), their attention is averaged, and
    the average is accumulated backward from the current position as in
    grouping_count. Returns (n_h, cum)."""
    P, n = Q.shape[0], K.shape[0]
    pbar = np.zeros(n, dtype=np.float64)
    for p in range(P):
        m = n - (P - 1 - p)
        pbar[:m] += attention_weights(Q[p], K[:m])
    pbar /= P
    cum = np.cumsum(pbar[::-1])
    hit = np.nonzero(cum >= tau)[0]
    n_h = int(hit[0]) + 1 if hit.size else int(cum.size)
    return n_h, cum


# Variant (not in the paper): distance on the image grid. Image token i sits
# in row i // row_len, column i % row_len (end-of-row tokens included); the
# distance of two image tokens is the squared Euclidean distance of their
# cells, an integer.
RASTER, GRID2D = 0, 1


def grid_d2(i: int, j: int, row_len: int) -> int:
    """Squared grid distance of image tokens i and j."""
    dr = i // row_len - j // row_len
    dc = i % row_len - j % row_len
    return dr * dr + dc * dc


def count_order_2d(n_tokens: int, n_cond: int, row_len: int) -> np.ndarray:
    """Order in which the 2D variant of Step 2 counts the tokens of a cache in
    position order (0 .. n_tokens-1, the first n_cond conditioning): image
    tokens by grid distance from the newest image token, nearest first, equal
    distances newer first; then the conditioning tokens, newest first (they
    have no cell and come last, as in the raster count)."""
    ref = n_tokens - 1 - n_cond
    img = sorted(range(n_cond, n_tokens),
                 key=lambda p: (grid_d2(p - n_cond, ref, row_len), -p))
    return np.array(img + list(range(n_cond - 1, -1, -1)), dtype=np.int64)


def _count_along(pbar, order, tau: float):
    cum = np.cumsum(pbar[order])
    hit = np.nonzero(cum >= tau)[0]
    n_h = int(hit[0]) + 1 if hit.size else int(cum.size)
    return n_h, cum


def grouping_count_2d(q, K, tau: float, n_cond: int, row_len: int):
    """Step 2 with the count running outward on the grid (count_order_2d)
    instead of backward in raster order. K holds the cache in position
    order. Returns (n_h, cum)."""
    p = attention_weights(q, K)
    return _count_along(p, count_order_2d(K.shape[0], n_cond, row_len), tau)


def grouping_count_multi_2d(Q, K, tau: float, n_cond: int, row_len: int):
    """grouping_count_multi's averaged attention counted in count_order_2d
    (outward from the current, newest, token)."""
    P, n = Q.shape[0], K.shape[0]
    pbar = np.zeros(n, dtype=np.float64)
    for p in range(P):
        m = n - (P - 1 - p)
        pbar[:m] += attention_weights(Q[p], K[:m])
    pbar /= P
    return _count_along(pbar, count_order_2d(n, n_cond, row_len), tau)


def classify(n_h: int, w_loc: int) -> int:
    """Local head iff fewer than w_loc tokens carry tau of the attention."""
    return LOCAL if n_h < w_loc else GLOBAL


def label_margin(cum: np.ndarray, tau: float, w_loc: int) -> float:
    """|mass of the newest w_loc-1 tokens - tau|: the distance of the label
    decision from its threshold (n_h < w_loc <=> that mass >= tau)."""
    n = min(w_loc - 1, cum.size)
    mass = float(cum[n - 1]) if n > 0 else 0.0
    return abs(mass - tau)


def count_margin(cum: np.ndarray, tau: float, n_h: int) -> float:
    """Distance of the count n_h from its own threshold: n_h is the minimum n
    with cum[n-1] >= tau, so it changes if cum[n_h-1] falls below tau or
    cum[n_h-2] reaches it. Returns min(cum[n_h-1] - tau, tau - cum[n_h-2]),
    over the terms that exist (the mass of zero tokens is 0), as absolute
    values."""
    terms = []
    if 1 <= n_h <= cum.size:
        terms.append(abs(float(cum[n_h - 1]) - tau))
    terms.append(abs(tau - (float(cum[n_h - 2]) if n_h >= 2 else 0.0)))
    return min(terms)


# ----------------------------------------------------------------------------
# Sec. 5.1: budgets
# ----------------------------------------------------------------------------
def global_budget(rho: Fraction, n_image: int) -> int:
    """Image tokens kept by a global head: rho * N, rounded down."""
    return math.floor(Fraction(rho) * n_image)


def head_budget(label: int, B_g: int, w: int) -> int:
    """Global heads keep B_g image tokens; local heads keep the recent w."""
    return B_g if label == GLOBAL else w


def redistributed_budgets(group_labels, B_g: int, w: int) -> np.ndarray:
    """Budget variant (not in the paper; aggregate-preserving): within one
    (sequence, layer) group of H heads, the image tokens the local heads do
    not use, (H - n_g)(B_g - w), go to its n_g global heads in equal shares,
    the remainder one token each to the global heads of lowest index, so the
    group keeps H * B_g image tokens as if every head had B_g. A group
    without global heads keeps the paper's budgets."""
    lab = np.asarray(group_labels).reshape(-1)
    glob = np.flatnonzero(lab == GLOBAL)
    budget = np.array([head_budget(int(x), B_g, w) for x in lab], dtype=np.int64)
    if glob.size == 0:
        return budget
    extra = (lab.size - glob.size) * (B_g - w)
    share, rem = divmod(extra, glob.size)
    budget[glob] += share
    budget[glob[:rem]] += 1
    return budget


def arena_layout(labels, n_cond: int, B_g: int, w: int, P: int, group: int = 0):
    """Per-head budget, capacity (C + budget + P buffered tokens) and the
    exclusive prefix sum of capacities (segment offsets, in tokens) for heads
    in the given order. group > 0: the redistributed budgets over
    consecutive groups of that many heads (one (sequence, layer) each).
    Returns (budget, cap, off, total)."""
    labels = np.asarray(labels).reshape(-1)
    if group > 0:
        budget = np.concatenate([redistributed_budgets(labels[i: i + group], B_g, w)
                                 for i in range(0, labels.size, group)]) if labels.size else \
            np.zeros(0, np.int64)
    else:
        budget = np.array([head_budget(int(x), B_g, w) for x in labels], dtype=np.int64)
    cap = n_cond + budget + P
    off = np.zeros_like(cap)
    if cap.size:
        off[1:] = np.cumsum(cap)[:-1]
    return budget, cap, off, int(cap.sum())


# ----------------------------------------------------------------------------
# Sec. 4: Stratified Token Eviction (Eqs. 5-6)
# ----------------------------------------------------------------------------
def ste_partition(T: int, r_s: float) -> int:
    """Eq. 5: C_long = H[:T r_s] (the oldest), C_near = H[T r_s:]."""
    return int(math.floor(float(T) * float(r_s)))


def ste_long_2d(hist, n_long: int, n_cond: int, row_len: int, t_ref: int) -> np.ndarray:
    """2D variant of Eq. 5 (not in the paper): the long-range subset is the
    n_long history tokens (positions `hist`) farthest on the grid from image
    token t_ref (the newest), equal distances older first. Boolean mask over
    hist."""
    hist = np.asarray(hist)
    key = sorted(range(hist.size),
                 key=lambda j: (-grid_d2(int(hist[j]) - n_cond, t_ref, row_len), int(hist[j])))
    mask = np.zeros(hist.size, dtype=bool)
    mask[key[:n_long]] = True
    return mask


def ste_scores_eq6(Q_past, Ck) -> np.ndarray:
    """Eq. 6 as printed: (1/P) 1^T (Q_past Ck^T / sqrt(d)), fp64."""
    Q = np.asarray(Q_past, dtype=np.float64)
    K = np.asarray(Ck, dtype=np.float64)
    return (Q @ K.T / math.sqrt(Q.shape[1])).mean(axis=0)


def ste_scores_fp32(Q_past, Ck) -> np.ndarray:
    """The ranking of Eq. 6 in the precision the eviction is decided in.

    The positive factor 1/(P sqrt d) does not change the ranking and is
    dropped. In fp32, with every product and sum rounded on its own:
      qbar[d] = q_0[d] + q_1[d] + ... (oldest query first),
      s_j     = (((0 + qbar[0] k_j[0]) + qbar[1] k_j[1]) + ...)  (d ascending).
    """
    Q = np.asarray(Q_past, dtype=np.float32)
    K = np.asarray(Ck, dtype=np.float32)
    qbar = np.zeros(Q.shape[1], dtype=np.float32)
    for p in range(Q.shape[0]):
        qbar = qbar + Q[p]
    s = np.zeros(K.shape[0], dtype=np.float32)
    for d in range(K.shape[1]):
        s = s + qbar[d] * K[:, d]
    return s


def ste_quotas(M: int, n_long: int, n_near: int):
    """M/2 evictions from each subset: floor(M/2) from the long-range subset
    and the rest from the near-range one; a subset smaller than its quota
    hands the excess to the other."""
    assert 0 <= M <= n_long + n_near
    m_long, m_near = M // 2, M - M // 2
    if m_long > n_long:
        m_near += m_long - n_long
        m_long = n_long
    if m_near > n_near:
        m_long += m_near - n_near
        m_near = n_near
    return m_long, m_near


def ste_evict(scores, positions, n_long: int, M: int) -> np.ndarray:
    """Boolean eviction mask over the T history tokens (oldest first): in each
    subset the quota of lowest-score tokens is evicted, equal scores evicting
    the older token first."""
    scores = np.asarray(scores)
    positions = np.asarray(positions)
    T = scores.shape[0]
    m_long, m_near = ste_quotas(M, n_long, T - n_long)
    evict = np.zeros(T, dtype=bool)
    for lo, hi, m in ((0, n_long, m_long), (n_long, T, m_near)):
        if m == 0:
            continue
        order = np.lexsort((positions[lo:hi], scores[lo:hi]))
        evict[lo + order[:m]] = True
    return evict


def ste_evict_strata(scores, positions, is_long, M: int) -> np.ndarray:
    """ste_evict with the long-range subset given as a mask over the history
    tokens (any membership): the quotas of ste_quotas, each subset's lowest
    scores evicted, equal scores older first."""
    scores = np.asarray(scores)
    positions = np.asarray(positions)
    is_long = np.asarray(is_long, dtype=bool)
    n_long = int(is_long.sum())
    m_long, m_near = ste_quotas(M, n_long, scores.size - n_long)
    evict = np.zeros(scores.size, dtype=bool)
    for members, m in ((np.flatnonzero(is_long), m_long), (np.flatnonzero(~is_long), m_near)):
        if m == 0:
            continue
        order = np.lexsort((positions[members], scores[members]))
        evict[members[order[:m]]] = True
    return evict


# ----------------------------------------------------------------------------
# Eqs. 2-4: head-aware cache update
# ----------------------------------------------------------------------------
@dataclass
class HeadParams:
    n_cond: int
    n_image: int
    recent_w: int
    local_w: int
    period: int
    group_at: int
    global_budget: int
    tau: float
    r_s: float
    row_len: int = 0
    distance: int = RASTER   # GRID2D: the grid-distance variants of Step 2 and Eq. 5

    @property
    def hist_budget(self) -> int:
        return self.global_budget - self.recent_w

    @classmethod
    def of(cls, w, distance: int = RASTER) -> "HeadParams":
        return cls(n_cond=w.n_cond, n_image=w.n_image, recent_w=w.recent_w,
                   local_w=w.w_loc, period=w.period, group_at=w.group_at,
                   global_budget=global_budget(w.rho, w.n_image), tau=w.tau, r_s=w.r_s,
                   row_len=w.row_len, distance=distance)


@dataclass
class UpdateRecord:
    t_last: int            # last image token appended before the update
    T: int                 # history candidates
    n_long: int
    evicted: np.ndarray    # evicted positions (sorted)
    pos: np.ndarray        # retained positions after the update
    long_pos: np.ndarray | None = None   # positions of the long-range subset


def cache_update(pos: np.ndarray, label: int, hp: HeadParams, q, k, t_last: int,
                 scores: str = "fp32") -> UpdateRecord:
    """One cache update of a head. pos lists the retained cache tokens, oldest
    first (conditioning tokens are 0..C-1, image token t is C+t). The image
    part splits into the recent window (the newest w) and the history (the
    older ones). Local heads: history dropped (Eq. 3). Global heads: if the
    history exceeds its budget B_g - w, STE evicts the excess (Eq. 4)."""
    C, w = hp.n_cond, hp.recent_w
    cond = pos[pos < C]
    img = pos[pos >= C]
    n_recent = min(w, img.size)
    hist, recent = img[: img.size - n_recent], img[img.size - n_recent:]
    T = int(hist.size)
    n_long = ste_partition(T, hp.r_s)
    if hp.distance == GRID2D:
        is_long = ste_long_2d(hist, n_long, C, hp.row_len, t_last)
    else:
        is_long = np.arange(T) < n_long
    if label == LOCAL:
        evicted, kept = hist, hist[:0]
    elif T > hp.hist_budget:
        M = T - hp.hist_budget
        P = hp.period
        Q_past = q[t_last - P + 1: t_last + 1]
        Ck = k[hist]
        s = ste_scores_fp32(Q_past, Ck) if scores == "fp32" else ste_scores_eq6(Q_past, Ck)
        if hp.distance == GRID2D:
            ev = ste_evict_strata(s, hist, is_long, M)
        else:
            ev = ste_evict(s, hist, n_long, M)
        evicted, kept = hist[ev], hist[~ev]
    else:
        evicted, kept = hist[:0], hist
    new_pos = np.concatenate([cond, kept, recent])
    return UpdateRecord(t_last=t_last, T=T, n_long=n_long, evicted=evicted, pos=new_pos,
                        long_pos=hist[is_long])


@dataclass
class HeadTrace:
    label: int = -1                 # label used for compression
    label_computed: int = -1        # label from the grouping rule
    n_h: int = -1
    margin: float = float("nan")
    outputs: dict = field(default_factory=dict)   # t -> o_t (fp64 [D])
    pos_at: dict = field(default_factory=dict)    # t -> positions attended at step t
    updates: list = field(default_factory=list)   # UpdateRecord per update
    final_pos: np.ndarray | None = None
    nbuf: int = 0


def run_head(hp: HeadParams, q, k, v, *, label: int | None = None, record=(),
             record_pos=(), stop_after: int | None = None, scores: str = "fp32") -> HeadTrace:
    """Generate image tokens 0..N-1 for one head (Steps 1-3).

    q [N, d] holds the image-token queries; k, v [C+N, d] the keys and values
    indexed by cache position. `label` overrides the grouping result (used to
    continue from the label the device chose on a declared near-tie). The
    attention output is kept for the steps in `record`, the positions the
    attention saw for those in `record_pos`. `stop_after` ends the run after
    that image token's attention.
    """
    C, N, P, E = hp.n_cond, hp.n_image, hp.period, hp.group_at
    record, record_pos = set(record), set(record_pos)
    tr = HeadTrace()
    pos = np.arange(C, dtype=np.int64)       # Step 1: cache of the condition
    compressed = False
    nbuf = 0
    last = N - 1 if stop_after is None else stop_after
    for t in range(last + 1):
        if compressed and nbuf == P:          # periodic update (buffer full)
            rec = cache_update(pos, tr.label, hp, q, k, t - 1, scores)
            tr.updates.append(rec)
            pos, nbuf = rec.pos, 0
        pos = np.append(pos, C + t)           # K <- [K, k_t], V <- [V, v_t]
        if compressed:
            nbuf += 1
        if t in record:
            tr.outputs[t] = attention(q[t], k[pos], v[pos])
        if t in record_pos:
            tr.pos_at[t] = pos.copy()
        if t == E - 1:                        # Step 2: head grouping
            if hp.distance == GRID2D:
                n_h, cum = grouping_count_2d(q[t], k[pos], hp.tau, C, hp.row_len)
            else:
                n_h, cum = grouping_count(q[t], k[pos], hp.tau)
            tr.n_h = n_h
            tr.label_computed = classify(n_h, hp.local_w)
            tr.margin = label_margin(cum, hp.tau, hp.local_w)
            tr.label = tr.label_computed if label is None else int(label)
            rec = cache_update(pos, tr.label, hp, q, k, t, scores)   # Step 3
            tr.updates.append(rec)
            pos, nbuf, compressed = rec.pos, 0, True
    tr.final_pos = pos
    tr.nbuf = nbuf
    return tr


def dense_causal_attention(q, k, v, n_cond: int) -> np.ndarray:
    """Full-cache attention of every image query over all tokens up to and
    including itself, as one masked matrix product (Eq. 1 with a causal
    mask): the uncompressed baseline the schedule must reproduce at full
    budget. Returns [N, d] fp64."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    N, d = q.shape
    logits = q @ k.T / math.sqrt(d)                     # [N, C+N]
    visible = np.arange(k.shape[0])[None, :] <= (n_cond + np.arange(N))[:, None]
    logits = np.where(visible, logits, -np.inf)
    logits -= logits.max(axis=1, keepdims=True)
    p = np.exp(logits)
    return (p @ v) / p.sum(axis=1, keepdims=True)
