"""InertiaKV oracle -- plain, slow, fp64 CPU restatement of the decode-step eviction loop.

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference legs of ``bench.py`` may import this package.  The
CUDA library never imports, links or calls it, and it shares no code with it.

What it computes, in the paper's order and notation (arxiv 2609.03515):

* Sec. 3, problem statement: a decode-side budget ``B`` per sequence; eviction
  is irreversible; whenever the cache exceeds ``B`` the tokens with the lowest
  utility ``m_t(i)`` are evicted.
* Eq. 1: per-step score ``s_t(i) = (1/H) sum_h a_t^(h)(i)``, where ``a_t^(h)`` is
  the last query's softmax attention of head ``h`` over the cached tokens.
* Eq. 4 + Appendix "Layer scoring": the EMA state is updated after every
  eligible layer, ``m_{t,l} = alpha m_{t,l-1} + (1-alpha) s_{t,l}``, with
  ``m_{t,0} = m_{t-1,K}``.
* Appendix "Momentum initialization": ``m_0 = 0``; no EMA during prefill.
* Eq. 6 (Lazy refresh): refresh steps ``R_r = {t >= 1 : (t-1) mod r = 0}``;
  off-refresh the state is carried unchanged and no attention score is taken.
* Score-Free box (Sec. 3.2): score at step 1 only, then freeze; eviction
  continues with the frozen ranking.
* Appendix "New token insertion during non-refresh steps": the new token's
  state is the mean of the existing tokens' state; it may be evicted at once.
* Appendix "Eviction on non-refresh steps": the stale state still drives
  eviction, so the budget always holds.

Readings taken where the paper is silent (each also stated where it is used):

* R1 (granularity): one state row per sequence, shared by every layer and KV
  head (``GRAN_SEQ``, Eq. 1 with ``m_t in R^{L_t}``).  ``GRAN_KVHEAD`` keeps one
  row per (sequence, KV head) whose score is the mean over that head's query
  group (Appendix "Per-step scoring", GQA sentence); its kept set applies to
  that KV head in every layer.
* R2 (eviction time): eviction happens once per step, after all layers, with
  the step's final state ``m_{t,K}``; the same kept set applies to every layer.
* R3 (new token on refresh steps): state 0 (as ``m_0 = 0``), then scored in
  the same step.  The mean rule applies on non-refresh steps only.
* R4 (ties): among equal utilities the lower cache slot is kept; ``-0.0``
  equals ``+0.0``; NaN ranks below every number.
* R5 (order): survivors keep their relative order (stable compaction); the
  appended token is last before eviction.
* R6 (self-attention): the appended token is part of its own step's softmax.
* R7 (scale): softmax scale ``1/sqrt(d)``; keys are used as stored.
* R8 (eligible layers): all layers unless a layer mask says otherwise.
* R10 (per-layer immediate eviction, the Appendix "Layer scoring" hook read
  literally): every layer, right after its own update of the state, evicts down
  to the budget from the tokens that layer holds, by the state as it stands then
  (m_{t,l}).  Layers then hold different token sets, so the state is indexed by
  token position and shared by all layers.  A layer's update covers every live
  position (held by at least one layer): a token the layer does not hold got no
  attention there, so its score is 0 (Eq. 1) and Eq. 4 decays it.  The new
  token's mean initialisation on non-refresh steps averages over the live
  positions.  With one layer this is the base method exactly.
* R11 (rank-trace diagnostics, Appendix "Mechanistic Diagnostics"): on every
  refresh step the raw top-k set R_t is the k = B tokens with the highest
  single-step score (Eq. 2: the last eligible layer's Eq. 1 score, i.e. the
  utility alpha = 0 would give), ties to the lower slot (R4), taken over the
  step's cache before eviction; the EMA top-k set E_t is the kept set.  Churn of
  a set is 1 - |X_t & X_{t'}| / |X_t| against the previous traced step t';
  raw/EMA Jaccard |R_t & E_t| / |R_t | E_t|; raw-top evicted 1 - |R_t & E_t| / |R_t|.
  Sets are compared by token position.
* R9 (scorer variants, Appendix "Per-step scoring"): VNorm divides each value
  row's l2 norm by the mean norm over the cached tokens of its (layer, KV head);
  entropy weighting uses the normalized entropy H(s) / ln n of the layer's
  pooled score distribution s over the n cached tokens (per utility row), and
  weight 1 when n = 1 or when a head's values are all zero.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

GRAN_SEQ = 0
GRAN_KVHEAD = 1


# --------------------------------------------------------------------------
# Attention and the per-step score (Eq. 1)
# --------------------------------------------------------------------------
def softmax(z: np.ndarray) -> np.ndarray:
    """Row softmax with the usual max shift (Vaswani et al., as cited for Eq. 1)."""
    z = np.asarray(z, dtype=np.float64)
    zmax = np.max(z, axis=-1, keepdims=True)
    e = np.exp(z - zmax)
    return e / np.sum(e, axis=-1, keepdims=True)


def last_query_attention(q: np.ndarray, K: Sequence[np.ndarray], V: Sequence[np.ndarray]):
    """Attention of one layer's last query over its cached tokens (Eq. 1's ``a_t^(h)``).

    q: [H, d] (the new token's query per head); K[g], V[g]: [L, d] per KV head.
    Query head h reads KV head ``h // (H / H_kv)`` (grouped-query attention).
    Returns (a [H, L] softmax probabilities, out [H, d] attention output).
    """
    q = np.asarray(q, dtype=np.float64)
    H, d = q.shape
    n_kv = len(K)
    group = H // n_kv
    L = K[0].shape[0]
    a = np.empty((H, L))
    out = np.empty((H, d))
    for h in range(H):
        g = h // group
        z = (np.asarray(K[g], np.float64) @ q[h]) / np.sqrt(d)
        a[h] = softmax(z)
        out[h] = a[h] @ np.asarray(V[g], np.float64)
    return a, out


def pooled_score(a: np.ndarray, granularity: int, kv_heads: int) -> np.ndarray:
    """Eq. 1: mean of the heads' probabilities per cached token.

    GRAN_SEQ -> [1, L], mean over all H heads.
    GRAN_KVHEAD -> [H_kv, L], mean over each KV head's query group (reading R1).
    """
    H, L = a.shape
    if granularity == GRAN_SEQ:
        return a.mean(axis=0, keepdims=True)
    return a.reshape(kv_heads, H // kv_heads, L).mean(axis=1)


def vnorm_weights(V_l: Sequence[np.ndarray]) -> np.ndarray:
    """Appendix "Per-step scoring", VNorm: for each KV head g, the l2 norm of every cached
    value row divided by the mean of those norms over the cached tokens.  [H_kv, L].
    (All-zero values of a head: weight 1, reading R9.)"""
    n = np.stack([np.sqrt(np.sum(np.asarray(v, np.float64) ** 2, axis=1)) for v in V_l])
    mean = n.mean(axis=1, keepdims=True)
    return np.where(mean > 0, n / np.where(mean > 0, mean, 1.0), 1.0)


def vnorm_score(a: np.ndarray, V_l: Sequence[np.ndarray], granularity: int, kv_heads: int) -> np.ndarray:
    """VNorm per-step score: each head's probabilities times its KV head's value-norm
    weights, then pooled as in Eq. 1."""
    H, L = a.shape
    w = vnorm_weights(V_l)
    return pooled_score(a * np.repeat(w, H // kv_heads, axis=0), granularity, kv_heads)


def entropy_weight(s_row: np.ndarray) -> float:
    """Entropy weighting: a layer's contribution is scaled by the normalized entropy of its
    pooled score distribution (which sums to 1 over the cached tokens), H(s) / ln n;
    1 when a single token is cached (reading R9)."""
    s_row = np.asarray(s_row, np.float64)
    n = s_row.size
    if n <= 1:
        return 1.0
    p = s_row[s_row > 0]
    return float(-np.sum(p * np.log(p)) / np.log(n))


# --------------------------------------------------------------------------
# Aggregation (Eq. 4, Appendix "Layer scoring")
# --------------------------------------------------------------------------
def ema_update(m: np.ndarray, s: np.ndarray, alpha: float) -> np.ndarray:
    """Eq. 4: m <- alpha m + (1 - alpha) s."""
    return alpha * m + (1.0 - alpha) * s


def cumulative_update(m: np.ndarray, s: np.ndarray) -> np.ndarray:
    """Eq. 3 (cumulative, H2O-style): m <- m + s."""
    return m + s


def single_step_update(m: np.ndarray, s: np.ndarray) -> np.ndarray:
    """Eq. 2 (single-step): m <- s."""
    return np.array(s, dtype=np.float64, copy=True)


def aggregate(m: np.ndarray, s: np.ndarray, p: "Params") -> np.ndarray:
    """One layer's update of the running utility under the configured rule (Eq. 2-4),
    applied after every eligible layer in the Appendix's layer-sequential order."""
    if p.aggregation == "ema":
        return ema_update(m, s, p.alpha)
    if p.aggregation == "cumulative":
        return cumulative_update(m, s)
    if p.aggregation == "single":
        return single_step_update(m, s)
    raise ValueError(p.aggregation)


def layer_sequential_ema(m_prev: np.ndarray, layer_scores: Sequence[np.ndarray], alpha: float) -> np.ndarray:
    """Appendix "Layer scoring": m_{t,0} = m_{t-1,K}; m_{t,l} = alpha m_{t,l-1} + (1-alpha) s_{t,l}."""
    m = np.array(m_prev, dtype=np.float64, copy=True)
    for s in layer_scores:
        m = ema_update(m, s, alpha)
    return m


# --------------------------------------------------------------------------
# Schedule (Eq. 6, Score-Free box)
# --------------------------------------------------------------------------
def is_refresh(t: int, refresh_period: int, score_free: bool) -> bool:
    """Eq. 6: t in R_r iff (t-1) mod r == 0 (t is 1-based).  Score-Free: t == 1 only."""
    if score_free:
        return t == 1
    return (t - 1) % refresh_period == 0


def new_token_state(m_row: np.ndarray, refresh: bool, refresh_init: str = "zero") -> float:
    """Utility given to the appended token.

    Non-refresh step: mean of the existing L_t - 1 tokens' state (Appendix "New
    token insertion", also the Score-Free box).  Refresh step: 0 (reading R3).
    """
    if refresh and refresh_init == "zero":
        return 0.0
    if m_row.size == 0:
        return 0.0
    return float(np.mean(m_row))


# --------------------------------------------------------------------------
# Budgeted selection (Sec. 3: evict the lowest m while the cache exceeds B)
# --------------------------------------------------------------------------
def select_keep(m_row: np.ndarray, budget: int) -> np.ndarray:
    """Kept slots, ascending: the ``budget`` highest utilities (ties: lower slot, R4).

    A full sort by (NaN last, m descending, slot ascending); no partial selection.
    """
    m_row = np.asarray(m_row, dtype=np.float64)
    L = m_row.shape[0]
    if L <= budget:
        return np.arange(L)
    nan = np.isnan(m_row)
    key = np.where(nan, -np.inf, m_row)
    order = np.lexsort((np.arange(L), -key, nan))
    return np.sort(order[:budget])


# --------------------------------------------------------------------------
# Cache state and one decode step
# --------------------------------------------------------------------------
@dataclass
class Params:
    alpha: float = 0.8                 # Sec. 3.1 default 0.8
    refresh_period: int = 1            # r of Eq. 6; 1 = full refresh
    score_free: bool = False
    granularity: int = GRAN_SEQ
    layer_mask: Optional[List[bool]] = None   # eligible layers (R8)
    refresh_init: str = "zero"         # R3
    aggregation: str = "ema"           # Eq. 4 (InertiaKV); "cumulative" (Eq. 3) or "single" (Eq. 2)
    scorer: str = "attention"          # Eq. 1; "vnorm" or "entropy" (Appendix "Per-step scoring")


@dataclass
class SeqState:
    """One sequence's cache: K[l][g], V[l][g] are [L, d]; m, pos are [R, L]."""

    K: List[List[np.ndarray]]
    V: List[List[np.ndarray]]
    m: np.ndarray
    pos: np.ndarray
    budget: int
    next_pos: int
    granularity: int = GRAN_SEQ
    raw: Optional[np.ndarray] = None   # [R, L] last eligible layer's score of the step (R11)

    @property
    def length(self) -> int:
        return self.m.shape[1]

    @property
    def layers(self) -> int:
        return len(self.K)

    @property
    def kv_heads(self) -> int:
        return len(self.K[0])

    def row_of(self, g: int) -> int:
        return 0 if self.granularity == GRAN_SEQ else g


def prefill_state(K: Sequence[Sequence[np.ndarray]], V: Sequence[Sequence[np.ndarray]], budget: int,
                  granularity: int = GRAN_SEQ) -> SeqState:
    """State after prefill: full cache, m_0 = 0 (Appendix "Momentum initialization")."""
    layers, kv = len(K), len(K[0])
    L0 = K[0][0].shape[0]
    R = 1 if granularity == GRAN_SEQ else kv
    return SeqState(
        K=[[np.array(K[l][g], np.float64) for g in range(kv)] for l in range(layers)],
        V=[[np.array(V[l][g], np.float64) for g in range(kv)] for l in range(layers)],
        m=np.zeros((R, L0)), pos=np.tile(np.arange(L0, dtype=np.int64), (R, 1)),
        budget=budget, next_pos=L0, granularity=granularity)


def append_token(st: SeqState, k_new: np.ndarray, v_new: np.ndarray, refresh: bool, p: Params) -> None:
    """Append the new token's K/V rows ([layers][kv_heads][d]) at the end of the cache."""
    R = st.m.shape[0]
    init = np.array([new_token_state(st.m[r], refresh, p.refresh_init) for r in range(R)])
    for l in range(st.layers):
        for g in range(st.kv_heads):
            st.K[l][g] = np.vstack([st.K[l][g], np.asarray(k_new[l][g], np.float64)[None]])
            st.V[l][g] = np.vstack([st.V[l][g], np.asarray(v_new[l][g], np.float64)[None]])
    st.m = np.concatenate([st.m, init[:, None]], axis=1)
    st.pos = np.concatenate([st.pos, np.full((R, 1), st.next_pos, np.int64)], axis=1)
    st.next_pos += 1


def attend_and_score(st: SeqState, q_t: np.ndarray, refresh: bool, p: Params) -> np.ndarray:
    """All layers' attention outputs [layers][H][d]; on refresh steps, the
    layer-sequential EMA of Eq. 1 scores over the eligible layers (Appendix "Layer scoring")."""
    outs = []
    for l in range(st.layers):
        if st.granularity == GRAN_SEQ:
            a, o = last_query_attention(q_t[l], st.K[l], st.V[l])
        else:
            # each KV head holds its own kept set; query group of head g reads it
            H = q_t[l].shape[0]
            group = H // st.kv_heads
            a_parts, o_parts = [], []
            for g in range(st.kv_heads):
                ag, og = last_query_attention(q_t[l][g * group:(g + 1) * group], [st.K[l][g]], [st.V[l][g]])
                a_parts.append(ag)
                o_parts.append(og)
            a, o = np.vstack(a_parts), np.vstack(o_parts)
        outs.append(o)
        eligible = p.layer_mask is None or p.layer_mask[l]
        if refresh and eligible:
            if p.scorer == "vnorm":
                s = vnorm_score(a, st.V[l], st.granularity, st.kv_heads)
            else:
                s = pooled_score(a, st.granularity, st.kv_heads)
            if p.scorer == "entropy":
                s = s * np.array([[entropy_weight(row)] for row in s])
            st.m = aggregate(st.m, s, p)
            st.raw = s
    return np.stack(outs)


def evict(st: SeqState, keep_override: Optional[Sequence[np.ndarray]] = None) -> List[np.ndarray]:
    """Evict down to the budget (Sec. 3), stable compaction (R5).  Returns kept slots per row."""
    R = st.m.shape[0]
    keeps = []
    for r in range(R):
        keep = select_keep(st.m[r], st.budget) if keep_override is None else np.asarray(keep_override[r])
        keeps.append(np.asarray(keep, np.int64))
    if st.length <= st.budget and keep_override is None:
        return keeps
    new_m = np.stack([st.m[r][keeps[r]] for r in range(R)])
    new_pos = np.stack([st.pos[r][keeps[r]] for r in range(R)])
    for l in range(st.layers):
        for g in range(st.kv_heads):
            kr = keeps[st.row_of(g)]
            st.K[l][g] = st.K[l][g][kr]
            st.V[l][g] = st.V[l][g][kr]
    st.m, st.pos = new_m, new_pos
    return keeps


def decode_step(st: SeqState, t: int, q_t: np.ndarray, k_new: np.ndarray, v_new: np.ndarray, p: Params) -> np.ndarray:
    """One decode step t (1-based) for one sequence; returns the attention outputs [layers][H][d].

    q_t: [layers][H][d]; k_new, v_new: [layers][H_kv][d].
    """
    refresh = is_refresh(t, p.refresh_period, p.score_free)
    st.raw = None
    append_token(st, k_new, v_new, refresh, p)
    out = attend_and_score(st, q_t, refresh, p)
    evict(st)
    return out


# --------------------------------------------------------------------------
# The same step for a sequence whose K/V rows are not held (workload sizes)
# --------------------------------------------------------------------------
@dataclass
class StreamState:
    """One sequence's eviction state without its cache: for every utility row r, the
    original token positions held, in slot order (``pos[r]``), and their utilities
    (``m[r]``).  A token's K/V rows never change (Sec. 3: eviction only removes tokens),
    so a step fetches the rows it needs by position instead of keeping them."""

    pos: np.ndarray
    m: np.ndarray
    budget: int
    next_pos: int
    layers: int
    kv_heads: int
    granularity: int = GRAN_SEQ
    raw: Optional[np.ndarray] = None

    @property
    def length(self) -> int:
        return self.m.shape[1]


def stream_prefill_state(L0: int, budget: int, layers: int, kv_heads: int,
                         granularity: int = GRAN_SEQ) -> StreamState:
    """State after prefill: positions 0..L0-1 in order, m_0 = 0 (Appendix "Momentum initialization")."""
    R = 1 if granularity == GRAN_SEQ else kv_heads
    return StreamState(pos=np.tile(np.arange(L0, dtype=np.int64), (R, 1)), m=np.zeros((R, L0)), budget=budget,
                       next_pos=L0, layers=layers, kv_heads=kv_heads, granularity=granularity)


def decode_step_streaming(st: StreamState, t: int, q_t: np.ndarray, kv_rows, p: Params,
                          keep_override=None) -> np.ndarray:
    """One decode step t (1-based) of one sequence, as ``decode_step``, with the cached
    rows fetched by position: ``kv_rows(l, g, positions)`` returns (K, V), each
    [len(positions), d], the rows of layer l / KV head g at those original positions
    (the appended token's position included).

    Steps in the paper's order: (1) append the new token at the end of every row, state 0
    on refresh steps (reading R3) or the mean of the row's existing states (Appendix "New
    token insertion"); (2) every layer's last-query attention over the row's tokens and, on
    refresh steps of an eligible layer, its Eq. 1 score (or the VNorm / entropy-weighted
    score) folded into the state in ascending layer order (Eq. 2-4, Appendix "Layer
    scoring"); (3) if the row holds more than B tokens, keep the B highest utilities (ties
    to the lower slot) in slot order (Sec. 3, R4, R5).

    keep_override(r, m_row, pos_row) may return the kept slots of row r (ascending)
    instead of the row's own top-B choice; it is called for every row after step (2),
    with the row's state as the selection sees it (lock-step tests).  Returns the
    attention outputs [layers][H][d]."""
    refresh = is_refresh(t, p.refresh_period, p.score_free)
    st.raw = None
    R = st.m.shape[0]
    # (1) append
    init = np.array([new_token_state(st.m[r], refresh, p.refresh_init) for r in range(R)])
    st.m = np.concatenate([st.m, init[:, None]], axis=1)
    st.pos = np.concatenate([st.pos, np.full((R, 1), st.next_pos, np.int64)], axis=1)
    st.next_pos += 1
    # (2) attention of every layer; the score and the layer-sequential update on refresh steps
    outs = []
    for l in range(st.layers):
        H = q_t[l].shape[0]
        group = H // st.kv_heads
        if st.granularity == GRAN_SEQ:
            rows = [kv_rows(l, g, st.pos[0]) for g in range(st.kv_heads)]
            K_l = [np.asarray(k, np.float64) for k, _ in rows]
            V_l = [np.asarray(v, np.float64) for _, v in rows]
            a, o = last_query_attention(q_t[l], K_l, V_l)
        else:
            # reading R1: KV head g holds its own tokens; its query group reads them
            a_parts, o_parts, V_l = [], [], []
            for g in range(st.kv_heads):
                k, v = kv_rows(l, g, st.pos[g])
                V_l.append(np.asarray(v, np.float64))
                ag, og = last_query_attention(q_t[l][g * group:(g + 1) * group], [np.asarray(k, np.float64)],
                                              [V_l[g]])
                a_parts.append(ag)
                o_parts.append(og)
            a, o = np.vstack(a_parts), np.vstack(o_parts)
        outs.append(o)
        eligible = p.layer_mask is None or p.layer_mask[l]
        if refresh and eligible:
            if p.scorer == "vnorm":
                s = vnorm_score(a, V_l, st.granularity, st.kv_heads)
            else:
                s = pooled_score(a, st.granularity, st.kv_heads)
            if p.scorer == "entropy":
                s = s * np.array([[entropy_weight(row)] for row in s])
            st.m = aggregate(st.m, s, p)
            st.raw = s
    # (3) eviction down to the budget, survivors in slot order
    keeps = []
    for r in range(R):
        keep = None if keep_override is None else keep_override(r, st.m[r].copy(), st.pos[r].copy())
        keeps.append(select_keep(st.m[r], st.budget) if keep is None else np.asarray(keep, np.int64))
    if st.length > st.budget or keep_override is not None:
        st.m = np.stack([st.m[r][keeps[r]] for r in range(R)])
        st.pos = np.stack([st.pos[r][keeps[r]] for r in range(R)])
    return np.stack(outs)


# --------------------------------------------------------------------------
# Per-layer immediate eviction (reading R10)
# --------------------------------------------------------------------------
@dataclass
class LayerwiseState:
    """One sequence under per-layer eviction: layer l holds the tokens pos[l] (ascending
    positions, slot order) with rows K[l][g], V[l][g] ([len(pos[l]), d]); m[p] is the
    shared state of position p (every position ever appended; only live ones matter)."""

    K: List[List[np.ndarray]]
    V: List[List[np.ndarray]]
    pos: List[np.ndarray]
    m: np.ndarray
    budget: int
    next_pos: int

    @property
    def layers(self) -> int:
        return len(self.K)

    @property
    def kv_heads(self) -> int:
        return len(self.K[0])

    def live(self) -> np.ndarray:
        """Positions held by at least one layer, ascending."""
        return np.unique(np.concatenate(self.pos))


def layerwise_prefill_state(K, V, budget: int) -> LayerwiseState:
    layers, kv = len(K), len(K[0])
    L0 = K[0][0].shape[0]
    return LayerwiseState(
        K=[[np.array(K[l][g], np.float64) for g in range(kv)] for l in range(layers)],
        V=[[np.array(V[l][g], np.float64) for g in range(kv)] for l in range(layers)],
        pos=[np.arange(L0, dtype=np.int64) for _ in range(layers)],
        m=np.zeros(L0), budget=budget, next_pos=L0)


@dataclass
class LayerTrace:
    """What layer l's eviction saw: its held positions and their state m_{t,l}."""
    pos: np.ndarray
    m: np.ndarray
    kept: np.ndarray


def decode_step_layerwise(st: LayerwiseState, t: int, q_t: np.ndarray, k_new: np.ndarray, v_new: np.ndarray,
                          p: Params, keep_override=None):
    """One decode step under per-layer immediate eviction (reading R10).

    q_t: [layers][H][d]; k_new, v_new: [layers][H_kv][d].  keep_override(l, trace) may
    return the positions layer l keeps instead of its own top-B choice (lock-step tests).
    Returns (attention outputs [layers][H][d], [LayerTrace per layer])."""
    refresh = is_refresh(t, p.refresh_period, p.score_free)
    # append: every layer gets the new token; its state is 0 on refresh steps (R3),
    # else the mean over the live positions (Appendix "New token insertion", R10)
    live = st.live()
    if refresh and p.refresh_init == "zero":
        init = 0.0
    else:
        init = float(np.mean(st.m[live])) if live.size else 0.0
    st.m = np.append(st.m, init)
    for l in range(st.layers):
        for g in range(st.kv_heads):
            st.K[l][g] = np.vstack([st.K[l][g], np.asarray(k_new[l][g], np.float64)[None]])
            st.V[l][g] = np.vstack([st.V[l][g], np.asarray(v_new[l][g], np.float64)[None]])
        st.pos[l] = np.append(st.pos[l], st.next_pos)
    st.next_pos += 1
    outs, traces = [], []
    for l in range(st.layers):
        a, o = last_query_attention(q_t[l], st.K[l], st.V[l])
        outs.append(o)
        eligible = p.layer_mask is None or p.layer_mask[l]
        if refresh and eligible:
            # Eq. 1 over the layer's own tokens; 0 for live positions it does not hold
            s_pos = np.zeros_like(st.m)
            s_pos[st.pos[l]] = pooled_score(a, GRAN_SEQ, st.kv_heads)[0]
            live = st.live()
            st.m[live] = ema_update(st.m[live], s_pos[live], p.alpha)
        m_l = st.m[st.pos[l]]
        keep = select_keep(m_l, st.budget)
        tr = LayerTrace(pos=st.pos[l].copy(), m=m_l.copy(), kept=st.pos[l][keep])
        if keep_override is not None:
            kp = keep_override(l, tr)
            if kp is not None:
                keep = np.searchsorted(st.pos[l], np.sort(np.asarray(kp, np.int64)))
                tr.kept = st.pos[l][keep]
        traces.append(tr)
        st.pos[l] = st.pos[l][keep]
        for g in range(st.kv_heads):
            st.K[l][g] = st.K[l][g][keep]
            st.V[l][g] = st.V[l][g][keep]
    return np.stack(outs), traces


@dataclass
class LayerwiseStreamState:
    """Per-layer eviction state of one sequence without its cache: the positions layer l
    holds, in slot order (``pos[l]``), and the state of every position appended so far
    (``m[p]``).  Rows are fetched by position when a step needs them."""

    pos: List[np.ndarray]
    m: np.ndarray
    budget: int
    next_pos: int
    kv_heads: int

    @property
    def layers(self) -> int:
        return len(self.pos)

    def live(self) -> np.ndarray:
        return np.unique(np.concatenate(self.pos))


def layerwise_stream_prefill_state(L0: int, budget: int, layers: int, kv_heads: int) -> LayerwiseStreamState:
    return LayerwiseStreamState(pos=[np.arange(L0, dtype=np.int64) for _ in range(layers)], m=np.zeros(L0),
                                budget=budget, next_pos=L0, kv_heads=kv_heads)


def decode_step_layerwise_streaming(st: LayerwiseStreamState, t: int, q_t: np.ndarray, kv_rows, p: Params,
                                    keep_override=None):
    """``decode_step_layerwise`` (reading R10) with every layer's rows fetched by position:
    ``kv_rows(l, g, positions)`` -> (K, V), each [len(positions), d].

    (1) every layer appends the new token; its state is 0 on refresh steps (R3), else the
    mean over the live positions; (2) layer by layer: attention over the layer's own
    tokens; on refresh steps of an eligible layer the Eq. 1 score (0 at live positions the
    layer does not hold) updates every live position by Eq. 4; then the layer keeps the B
    highest states among its tokens (ties to the lower slot), in slot order.
    keep_override(l, LayerTrace) as in ``decode_step_layerwise``.
    Returns (attention outputs [layers][H][d], [LayerTrace per layer])."""
    refresh = is_refresh(t, p.refresh_period, p.score_free)
    live = st.live()
    if refresh and p.refresh_init == "zero":
        init = 0.0
    else:
        init = float(np.mean(st.m[live])) if live.size else 0.0
    st.m = np.append(st.m, init)
    for l in range(st.layers):
        st.pos[l] = np.append(st.pos[l], st.next_pos)
    st.next_pos += 1
    outs, traces = [], []
    for l in range(st.layers):
        rows = [kv_rows(l, g, st.pos[l]) for g in range(st.kv_heads)]
        a, o = last_query_attention(q_t[l], [np.asarray(k, np.float64) for k, _ in rows],
                                    [np.asarray(v, np.float64) for _, v in rows])
        outs.append(o)
        eligible = p.layer_mask is None or p.layer_mask[l]
        if refresh and eligible:
            s_pos = np.zeros_like(st.m)
            s_pos[st.pos[l]] = pooled_score(a, GRAN_SEQ, st.kv_heads)[0]
            live = st.live()
            st.m[live] = ema_update(st.m[live], s_pos[live], p.alpha)
        m_l = st.m[st.pos[l]]
        keep = select_keep(m_l, st.budget)
        tr = LayerTrace(pos=st.pos[l].copy(), m=m_l.copy(), kept=st.pos[l][keep])
        if keep_override is not None:
            kp = keep_override(l, tr)
            if kp is not None:
                keep = np.searchsorted(st.pos[l], np.sort(np.asarray(kp, np.int64)))
                tr.kept = st.pos[l][keep]
        traces.append(tr)
        st.pos[l] = st.pos[l][keep]
    return np.stack(outs), traces


# --------------------------------------------------------------------------
# Rank-trace diagnostics (reading R11)
# --------------------------------------------------------------------------
def topk_positions(score_row: np.ndarray, pos_row: np.ndarray, k: int) -> np.ndarray:
    """Positions of the k highest scores of one row (ties: lower slot), ascending."""
    return np.sort(np.asarray(pos_row)[select_keep(score_row, k)])


def churn(cur: np.ndarray, prev: np.ndarray) -> float:
    """Fraction of a top-k set replaced since the previous traced step."""
    cur = set(np.asarray(cur).tolist())
    return 1.0 - len(cur & set(np.asarray(prev).tolist())) / len(cur) if cur else 0.0


def jaccard(a: np.ndarray, b: np.ndarray) -> float:
    a, b = set(np.asarray(a).tolist()), set(np.asarray(b).tolist())
    return len(a & b) / len(a | b) if a | b else 1.0


def raw_top_evicted(raw: np.ndarray, kept: np.ndarray) -> float:
    """Fraction of the raw top-k tokens not in the kept set."""
    raw = set(np.asarray(raw).tolist())
    return 1.0 - len(raw & set(np.asarray(kept).tolist())) / len(raw) if raw else 0.0


def decode_step_traced(st: SeqState, t: int, q_t, k_new, v_new, p: Params):
    """decode_step plus the step's rank-trace sets per row (R11): (out, [(R_t or None, E_t)])."""
    refresh = is_refresh(t, p.refresh_period, p.score_free)
    st.raw = None
    append_token(st, k_new, v_new, refresh, p)
    out = attend_and_score(st, q_t, refresh, p)
    R = [None if st.raw is None else topk_positions(st.raw[r], st.pos[r], st.budget) for r in range(st.m.shape[0])]
    evict(st)
    return out, [(R[r], np.sort(st.pos[r])) for r in range(st.m.shape[0])]
