"""fp64 CPU oracle of EpiKV's eviction path (test infrastructure only).

This module is test infrastructure.  Only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline leg may import it; the product path (the CUDA
library and its binding) never does, and shares no code with it.

It is a plain, slow, obviously correct restatement of the paper's definitions
in float64 with numpy: no blocking, fusion or reordering beyond what each
definition states.  Each function names the passage it follows.

Readings of points the paper leaves open (labels match the design notes):

R1  band combination: per-layer z-scores averaged within each band, Band A
    mean minus Band B mean; the singleton bands {10}, {21} give z10 - z21.
R2  z window: the last min(w, t) values g(t') with 1 <= t' <= t (causal,
    includes t; position 0 has no predecessor so no g); z(0) := 0.
R3  standard deviation is the population one (ddof 0); one value gives 0.
R4  eps = 1e-6 for both the z-score and the Lag-KV normalisation.
R5  the z numerator is the raw g_l(t) (Eq. 3), not the rolling mean.
R6  scores are computed once when a token is generated and then frozen.
R7  budget K counts every kept token: prefill + recency window + the top
    candidates; recency R = min(cap, floor(K / 4)) with cap = 128.  When
    prefill + R >= K the window shrinks to max(0, K - P); prefill is never
    evicted, so if P > K all P prefill tokens are kept.
R8  ties between equal scores go to the lower slot (earlier position); NaN
    ranks below every number; -0 equals +0.
R9  kept tokens stay in ascending position order after compaction.
R10 Lag-KV: chunks of lag positions at fixed boundaries t = c*lag; token t in
    chunk c >= 1 is normalised by the per-channel min/max over all positions
    of chunk c-1; population variance over the head dimension; K and V
    variances are added; the mean is over (layer, head); u(t) = 0 in chunk 0;
    the score is the mean of u over the last min(w, t+1) positions <= t.
R11 HS-variance (Eq. 2): the rolling mean of g over the same window as the
    z-score (R2); band means as in R1; s(0) = 0.
R12 KV-key / KV-val variance: the population variance over the head
    dimension of the stored key (value) vector of each (layer, head), mean
    over (layer, head), then the rolling mean of R10; every position has a
    value (no chunk 0 exception).
R13 lag-kv-key: Lag-KV (R10) with the key term only.
R18 chunk-level selection (named as future work in Sec. 5, after ChunkKV's
    contiguous chunks of Sec. 2): positions fall into fixed chunks
    floor(pos / C); a chunk's score is the mean of the frozen scores of its
    members that are candidates (prefill and recency slots are not members),
    here in float64 (a correctly rounded sum divided by the count); chunks
    rank by that score (R8's order: NaN lowest, -0 == +0, ties to the
    earlier chunk) and fill the M candidate places whole, in rank order; the
    first chunk that does not fit gives its lowest slots.  C = 1 is R7/R8.
R19 per-layer budgets (named as future work in Sec. 5, after PyramidKV's
    per-layer allocation of Sec. 2): layer l has its own budget K_l and its
    own cache, and evicts it by R7/R8 on its own, except that every layer
    uses the same recency window R = min(cap, floor(K_min / 4)), shrunk to
    max(0, K_min - P), K_min the smallest budget, and M_l = max(0, K_l - P -
    R); all layers evict at the same events, when the largest cache holds
    more than the trigger and more than K_min.  Equal budgets give R7.
"""
from __future__ import annotations

import math

import numpy as np

Z_EPS = 1e-6
LAG_EPS = 1e-6


# --------------------------------------------------------------------------
# Sec. 3.2, Eq. 1 -- hidden-state change
# --------------------------------------------------------------------------
def hidden_change(h_prev, h):
    """g = || h(t) - h(t-1) ||_2 for one pair of rows (Eq. 1)."""
    d = np.asarray(h, dtype=np.float64) - np.asarray(h_prev, dtype=np.float64)
    return float(np.sqrt(np.sum(d * d)))


def hidden_change_trace(rows):
    """g[t] for t = 1..T-1 of one layer's rows [T, D]; g[0] is NaN (Eq. 1)."""
    rows = np.asarray(rows, dtype=np.float64)
    g = np.full(rows.shape[0], np.nan)
    for t in range(1, rows.shape[0]):
        g[t] = hidden_change(rows[t - 1], rows[t])
    return g


# --------------------------------------------------------------------------
# Sec. 3.2, Eq. 3 -- causal rolling z-score
# --------------------------------------------------------------------------
def window_zscore(window, eps=Z_EPS):
    """(g(t) - mu) / (sigma + eps) over a trailing window whose last entry is
    g(t) (Eq. 3, readings R3-R5)."""
    w = np.asarray(window, dtype=np.float64)
    mu = np.mean(w)
    sigma = np.sqrt(np.mean((w - mu) ** 2))
    return float((w[-1] - mu) / (sigma + eps))


def rolling_zscore(g, w=64, eps=Z_EPS):
    """z[t] for a trace of g values indexed by position (Eq. 3, reading R2)."""
    g = np.asarray(g, dtype=np.float64)
    z = np.zeros(g.shape[0])
    for t in range(1, g.shape[0]):
        z[t] = window_zscore(g[max(1, t - w + 1): t + 1], eps)
    return z


def epiphany_score(z_band_a, z_band_b):
    """s = mean_{l in A} z_l - mean_{l in B} z_l (Eq. 3 combination, Fig. 1,
    reading R1).  Arguments are sequences of per-layer z arrays."""
    za = np.mean(np.asarray(z_band_a, dtype=np.float64), axis=0)
    zb = np.mean(np.asarray(z_band_b, dtype=np.float64), axis=0)
    return za - zb


def rolling_band_mean(g, w=64):
    """g-bar[t]: mean of g over the trailing window of R2 (Eq. 2); 0 at t = 0."""
    g = np.asarray(g, dtype=np.float64)
    m = np.zeros(g.shape[0])
    for t in range(1, g.shape[0]):
        m[t] = np.mean(g[max(1, t - w + 1): t + 1])
    return m


def hsvar_scores(rows_a, rows_b, w=64):
    """HS-variance score s(t) = g-bar_A(t) - g-bar_B(t) (Eq. 2, Tab. 1,
    reading R11) of every position of one sequence."""
    ma = [rolling_band_mean(hidden_change_trace(r), w) for r in rows_a]
    mb = [rolling_band_mean(hidden_change_trace(r), w) for r in rows_b]
    return np.mean(ma, axis=0) - np.mean(mb, axis=0)


def bandz_scores(rows_a, rows_b, w=64, eps=Z_EPS):
    """EpiKV score of every position 0..T-1 of one sequence.

    rows_a / rows_b: lists of [T, D] arrays, one per Band A / Band B layer.
    """
    za = [rolling_zscore(hidden_change_trace(r), w, eps) for r in rows_a]
    zb = [rolling_zscore(hidden_change_trace(r), w, eps) for r in rows_b]
    return epiphany_score(za, zb)


# --------------------------------------------------------------------------
# Sec. 3.3 -- Lag-KV: lag-normalised key+value variance
# --------------------------------------------------------------------------
def lag_token_variance(k_t, v_t, k_prev_chunk, v_prev_chunk, eps=LAG_EPS):
    """u(t) for one token whose chunk has a predecessor (Sec. 3.3, R10).

    k_t, v_t: [L, H, d] rows of the token; k_prev_chunk, v_prev_chunk:
    [lag, L, H, d] rows of every position of the previous chunk.
    """
    total = None
    for x, prev in ((k_t, k_prev_chunk), (v_t, v_prev_chunk)):
        x = np.asarray(x, dtype=np.float64)
        prev = np.asarray(prev, dtype=np.float64)
        mn = prev.min(axis=0)
        mx = prev.max(axis=0)
        xn = (x - mn) / (mx - mn + eps)                   # per-channel range
        mu = xn.mean(axis=-1, keepdims=True)
        var = ((xn - mu) ** 2).mean(axis=-1)              # over head dim, [L, H]
        total = var if total is None else total + var     # key + value
    return float(total.mean())                            # over (layer, head)


def head_variance(x):
    """mean over (layer, head) of the population variance over the head
    dimension of one token's stored vectors x [L, H, d] (Sec. 3.3, KV-key /
    KV-val, reading R12)."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    return float(((x - mu) ** 2).mean(axis=-1).mean())


def kv_variance_scores(X, w=64):
    """KV-key (X = keys) or KV-val (X = values) scores: the rolling mean of
    the per-token head variance (Sec. 3.3, Tab. 1, R12)."""
    return rolling_mean(np.array([head_variance(X[t]) for t in range(X.shape[0])]), w)


def lag_key_token_variance(k_t, k_prev_chunk, eps=LAG_EPS):
    """The key term of Lag-KV for one token (reading R13)."""
    x = np.asarray(k_t, dtype=np.float64)
    prev = np.asarray(k_prev_chunk, dtype=np.float64)
    mn = prev.min(axis=0)
    mx = prev.max(axis=0)
    xn = (x - mn) / (mx - mn + eps)
    return float(((xn - xn.mean(axis=-1, keepdims=True)) ** 2).mean(axis=-1).mean())


def lag_key_scores(K, lag=16, eps=LAG_EPS, w=64):
    """lag-kv-key scores: rolling mean of the key-only Lag-KV term (R13)."""
    T = K.shape[0]
    u = np.zeros(T)
    for t in range(lag, T):
        c = t // lag
        u[t] = lag_key_token_variance(K[t], K[(c - 1) * lag: c * lag], eps)
    return rolling_mean(u, w)


def lag_variance_trace(K, V, lag=16, eps=LAG_EPS):
    """u[t] for t = 0..T-1 from K, V rows [T, L, H, d]; u = 0 in chunk 0."""
    T = K.shape[0]
    u = np.zeros(T)
    for t in range(lag, T):
        c = t // lag
        lo, hi = (c - 1) * lag, c * lag
        u[t] = lag_token_variance(K[t], V[t], K[lo:hi], V[lo:hi], eps)
    return u


def rolling_mean(u, w=64):
    """Causal rolling mean over the last min(w, t+1) positions <= t (R10)."""
    u = np.asarray(u, dtype=np.float64)
    return np.array([np.mean(u[max(0, t - w + 1): t + 1]) for t in range(u.shape[0])])


def lagkv_scores(K, V, lag=16, eps=LAG_EPS, w=64):
    return rolling_mean(lag_variance_trace(K, V, lag, eps), w)


# --------------------------------------------------------------------------
# Sec. 3.1, Sec. 3.3 and App. D -- top-K retention under the budget
# --------------------------------------------------------------------------
def recency_window(K, cap=128):
    """R = min(128, K/4) (App. D)."""
    return min(cap, K // 4)


def select_kept(scores, K, prefill=0, recency_cap=128):
    """Ascending kept slot list of one sequence's cache (Sec. 3.1, App. D).

    scores[i] is the frozen score of cache slot i (slots are in position
    order).  Prefill slots and the trailing recency window are always kept;
    the remaining budget goes to the highest-scoring other slots (R7, R8).
    """
    scores = np.asarray(scores, dtype=np.float64)
    n = scores.shape[0]
    if n <= K:
        return list(range(n))
    P = min(prefill, n)
    R = min(recency_window(K, recency_cap), max(0, K - P))
    M = max(0, K - P - R)
    candidates = list(range(P, n - R))

    def rank(i):  # NaN last, higher score first, lower slot first
        s = scores[i]
        return (1, 0.0, i) if np.isnan(s) else (0, -s, i)

    best = sorted(candidates, key=rank)[:M]          # a full sort, no shortcuts
    kept = set(range(P)) | set(range(n - R, n)) | set(best)
    return sorted(kept)


def chunk_mean(values):
    """Mean of a chunk's member scores (R18): float64, the sum correctly
    rounded (NaN if any member is NaN)."""
    values = [float(v) for v in values]
    if any(math.isnan(v) for v in values):
        return float("nan")
    return math.fsum(values) / len(values)


def chunk_scores(scores, positions, candidates, chunk, mean=chunk_mean):
    """Mean score of every chunk of candidate slots (R18).

    Returns {chunk id: (mean, [member slots in slot order])}; chunk id =
    floor(position / chunk).  ``mean`` maps the members' scores (in slot
    order) to the chunk's score.
    """
    members = {}
    for i in candidates:
        members.setdefault(int(positions[i]) // chunk, []).append(i)
    return {c: (mean([scores[i] for i in slots]), slots) for c, slots in members.items()}


def select_kept_chunked(scores, positions, K, prefill=0, recency_cap=128, chunk=1, mean=chunk_mean):
    """Ascending kept slot list under chunk-level selection (R18).

    Same protected set and budget split as ``select_kept``; the M candidate
    places go to whole position chunks in the order of their mean score,
    the first chunk that does not fit contributing its lowest slots.
    """
    scores = np.asarray(scores, dtype=np.float64)
    n = scores.shape[0]
    if n <= K:
        return list(range(n))
    P = min(prefill, n)
    R = min(recency_window(K, recency_cap), max(0, K - P))
    M = max(0, K - P - R)
    candidates = list(range(P, n - R))
    chunks = chunk_scores(scores, positions, candidates, chunk, mean)

    def rank(c):  # NaN last, higher mean first, earlier chunk first
        s = float(chunks[c][0])
        return (1, 0.0, c) if np.isnan(s) else (0, -s, c)

    best = []
    for c in sorted(chunks, key=rank):
        slots = chunks[c][1]
        take = min(len(slots), M - len(best))
        best.extend(slots[:take])
        if len(best) == M:
            break
    kept = set(range(P)) | set(range(n - R, n)) | set(best)
    return sorted(kept)


def layer_recency(budgets, prefill, n, recency_cap=128):
    """The recency window every layer keeps under per-layer budgets (R19)."""
    k_min = min(budgets)
    P = min(prefill, n)
    return min(recency_window(k_min, recency_cap), max(0, k_min - P))


def select_kept_layer(scores, K, prefill, R):
    """One layer's ascending kept slot list of its own cache (R19): prefill,
    the last R slots and the K - P - R best other slots (R8 order)."""
    scores = np.asarray(scores, dtype=np.float64)
    n = scores.shape[0]
    P = min(prefill, n)
    assert n >= P + R, "a layer holds the prefill and the recency window"
    M = max(0, K - P - R)
    candidates = list(range(P, n - R))

    def rank(i):  # NaN last, higher score first, lower slot first
        s = scores[i]
        return (1, 0.0, i) if np.isnan(s) else (0, -s, i)

    best = sorted(candidates, key=rank)[:M]
    return sorted(set(range(P)) | set(range(n - R, n)) | set(best))


def simulate_decode_layers(scores, length, chunk, budgets, trigger, prefill=0, recency_cap=128):
    """Per-layer budgets (R19): every layer keeps its own cache of positions,
    appends ``chunk`` tokens at a time and, whenever the largest cache holds
    more than ``trigger`` tokens, evicts its own cache with its own budget.

    Returns the events as [(per-layer positions before, after)] and the final
    per-layer position lists.
    """
    caches = [[] for _ in budgets]
    events = []
    for start in range(0, length, chunk):
        new = list(range(start, min(length, start + chunk)))
        for c in caches:
            c.extend(new)
        n = max(len(c) for c in caches)
        if n > trigger and n > min(budgets):        # some layer is over its budget
            R = layer_recency(budgets, prefill, n, recency_cap)
            before = [list(c) for c in caches]
            caches = [[c[i] for i in select_kept_layer([scores[p] for p in c], K, prefill, R)]
                      for c, K in zip(caches, budgets)]
            events.append((before, [list(c) for c in caches]))
    return events, caches


# --------------------------------------------------------------------------
# App. H -- rebuild the cache from the kept entries, in order
# --------------------------------------------------------------------------
def compact(rows, kept):
    """Cache rows after eviction: the kept slots' rows, in slot order."""
    return np.asarray(rows)[np.asarray(kept, dtype=np.int64)]


def simulate_decode(scores, length, chunk, K, trigger, prefill=0, recency_cap=128, select_chunk=1):
    """Replay one sequence's decode: append ``chunk`` tokens at a time and
    evict whenever the cache holds more than ``trigger`` tokens.

    scores: frozen score of every position (R6).  ``select_chunk`` > 1 uses
    chunk-level selection (R18).  Returns the list of events as (positions
    before, positions after) and the final position list.
    """
    cache = []
    events = []
    for start in range(0, length, chunk):
        cache.extend(range(start, min(length, start + chunk)))
        if len(cache) > trigger:
            if select_chunk > 1:
                kept = select_kept_chunked([scores[p] for p in cache], cache, K, prefill, recency_cap,
                                           select_chunk)
            else:
                kept = select_kept([scores[p] for p in cache], K, prefill, recency_cap)
            after = [cache[i] for i in kept]
            events.append((list(cache), after))
            cache = list(after)
    return events, cache
