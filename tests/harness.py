"""Drives the CUDA library through its C ABI on seeded synthetic traces and
checks every stage against the fp64 oracle (test infrastructure).

Acceptance rules:
* scores: |s_gpu - s_ref| <= 1e-4 * max(1, |s_ref|), or, for the band-z
  score at a position whose z windows are ill-conditioned, <= 2u * kappa(t):
  u = 2^-24 is the fp32 unit roundoff of g and kappa(t) the score's
  sensitivity to relative perturbations of the g values (computed by
  bandz_condition from the oracle's own fp64 windows).  kappa is ~360 on the
  workloads (2u * kappa ~ 4e-5, so 1e-4 applies); it grows without bound when
  a window's g values nearly coincide (sigma << g), where no fp32 g can give
  the score to 1e-4;
* kept sets: the oracle's selection run on the GPU's own fp32 scores must
  equal the GPU's kept list exactly; against the oracle's fp64 scores, a slot
  may differ only if its reference score is within the score tolerance of the
  M-th candidate's score (a threshold tie); under chunk-level selection the
  same holds for the slot's chunk mean and the boundary chunk's mean;
* compacted K/V: byte-identical to the generator's rows of the kept positions.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from paper_2606_26472_gb300.cache import KVCache
from synth import gen, host
from synth.device import DeviceTrace, as_u16

TOL = 1e-4
U32 = 2.0 ** -24      # fp32 unit roundoff
ALL_KINDS = (E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV, E.EPIKV_SCORE_HSVAR, E.EPIKV_SCORE_KVKEY,
             E.EPIKV_SCORE_KVVAL, E.EPIKV_SCORE_LAGKEY)
BAND_KINDS = E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_HSVAR
KV_KINDS = E.EPIKV_SCORE_LAGKV | E.EPIKV_SCORE_KVKEY | E.EPIKV_SCORE_KVVAL | E.EPIKV_SCORE_LAGKEY


def score_bound(ref, cond=None):
    """Allowed |s_gpu - s_ref| per position (see the module docstring)."""
    ref = np.asarray(ref, dtype=np.float64)
    bound = TOL * np.maximum(1.0, np.abs(ref))
    if cond is not None:
        bound = np.maximum(bound, 2.0 * U32 * np.asarray(cond, dtype=np.float64))
    return bound


def bandz_condition_g(g_a, g_b, w=64, eps=O.Z_EPS):
    """kappa(t) of the band-z score from the band layers' g traces (g[0]
    unused): the sum over band layers of the band weight (1/|A| or 1/|B|)
    times (1 + |z_l(t)|) * max(window) / (sigma_l(t) + eps), a first-order
    bound of the score's change per unit relative error of the window's g."""
    T = len(g_a[0])
    kappa = np.zeros(T)
    for band, wt in ((g_a, 1.0 / len(g_a)), (g_b, 1.0 / len(g_b))):
        for g in band:
            for t in range(1, T):
                win = np.asarray(g[max(1, t - w + 1):t + 1], dtype=np.float64)
                mu = win.mean()
                sd = np.sqrt(np.mean((win - mu) ** 2))
                z = (g[t] - mu) / (sd + eps)
                kappa[t] += wt * (1.0 + abs(z)) * win.max() / (sd + eps)
    return kappa


def bandz_condition(rows_a, rows_b, w=64, eps=O.Z_EPS):
    """kappa(t) of the band-z score from the band layers' hidden rows."""
    return bandz_condition_g([O.hidden_change_trace(r) for r in rows_a],
                             [O.hidden_change_trace(r) for r in rows_b], w, eps)


def assert_scores_close(gpu, ref, what="", cond=None):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    bound = score_bound(ref, cond)
    bad = np.nonzero(~(np.abs(gpu - ref) <= bound))[0]
    if bad.size:
        i = bad[0]
        raise AssertionError(f"{what}: {bad.size} scores out of tolerance, first at {i}: gpu {gpu[i]!r} ref {ref[i]!r}")


ROW_BLOCK = 2048      # positions generated at a time by the oracle's traces (bounds host memory)


def band_g_trace(model, tabs, seq, layer, length, seg):
    """g_l(t) of one band layer for t < length (g[0] is NaN), Eq. 1: the
    oracle's hidden_change_trace over blocks of the generator's rows (each
    block starts one row early so that its first g has its predecessor)."""
    g = np.full(length, np.nan)
    for a in range(0, length, ROW_BLOCK):
        lo, b = max(0, a - 1), min(length, a + ROW_BLOCK)
        rows = gen.bf16_bits_to_f64(host.hidden_rows(model, tabs, seq, layer, np.arange(lo, b), seg))
        g[lo + 1:b] = O.hidden_change_trace(rows)[1:]
    return g


def kv_u_traces(model, tabs, seq, length, kinds, lag):
    """Per-position inputs of the K/V scores' rolling means (Sec. 3.3, R10,
    R12, R13): {kind: u[0..length)}, each u(t) from the oracle's per-token
    functions on the generator's rows of t and of its previous lag chunk,
    generated a block of positions at a time."""
    sp = gen.spike_flags(model, seq, length)
    u = {k: np.zeros(length) for k in ALL_KINDS if kinds & k & KV_KINDS}
    for a in range(0, length, ROW_BLOCK):
        b = min(length, a + ROW_BLOCK)
        first = max(0, (a // lag - 1) * lag)            # the previous chunk of a's chunk
        pos = np.arange(first, b)
        K = gen.bf16_bits_to_f64(host.kv_rows(model, tabs, seq, 0, pos, sp))
        V = gen.bf16_bits_to_f64(host.kv_rows(model, tabs, seq, 1, pos, sp))
        for t in range(a, b):
            i, c = t - first, t // lag
            lo = (c - 1) * lag - first
            if E.EPIKV_SCORE_KVKEY in u:
                u[E.EPIKV_SCORE_KVKEY][t] = O.head_variance(K[i])
            if E.EPIKV_SCORE_KVVAL in u:
                u[E.EPIKV_SCORE_KVVAL][t] = O.head_variance(V[i])
            if c == 0:
                continue                                   # u = 0 in chunk 0 (R10)
            if E.EPIKV_SCORE_LAGKV in u:
                u[E.EPIKV_SCORE_LAGKV][t] = O.lag_token_variance(K[i], V[i], K[lo:lo + lag], V[lo:lo + lag])
            if E.EPIKV_SCORE_LAGKEY in u:
                u[E.EPIKV_SCORE_LAGKEY][t] = O.lag_key_token_variance(K[i], K[lo:lo + lag])
    return u


class _LazyCond:
    """{kind: kappa[0..length)} of the band-z score, computed on first use."""

    def __init__(self, trace):
        self._t = trace
        self._v = None

    def _value(self):
        if self._v is None:
            t = self._t
            self._v = bandz_condition_g(t.g_a, t.g_b, t.z_window)
        return self._v

    def get(self, kind, default=None):
        return self._value() if kind == E.EPIKV_SCORE_BANDZ and self._t.has_bandz else default

    def __getitem__(self, kind):
        v = self.get(kind)
        if v is None:
            raise KeyError(kind)
        return v


class OracleTrace:
    """fp64 oracle scores of one sequence, positions 0..length-1, from the
    generator's rows (regenerated block by block by the host twin).

    Band kinds: every band layer's g trace (Eq. 1), then the oracle's rolling
    z-score and band combination (Eq. 3) or rolling band mean (Eq. 2).  K/V
    kinds: u(t) per position (Sec. 3.3), then the oracle's rolling mean."""

    def __init__(self, model, tabs, seq, length, kinds, z_window=64, lag=16, lag_window=64):
        self.length = length
        self.z_window = z_window
        self.scores = {}
        self.has_bandz = bool(kinds & E.EPIKV_SCORE_BANDZ)
        self.cond = _LazyCond(self)   # per-position sensitivity of the band-z score to fp32 rounding of g
        if kinds & BAND_KINDS:
            seg = gen.segment_index(model, seq, length)
            self.g_a = [band_g_trace(model, tabs, seq, l, length, seg) for l in model.band_a]
            self.g_b = [band_g_trace(model, tabs, seq, l, length, seg) for l in model.band_b]
            if kinds & E.EPIKV_SCORE_BANDZ:
                self.scores[E.EPIKV_SCORE_BANDZ] = O.epiphany_score(
                    [O.rolling_zscore(g, z_window) for g in self.g_a], [O.rolling_zscore(g, z_window) for g in self.g_b])
            if kinds & E.EPIKV_SCORE_HSVAR:
                self.scores[E.EPIKV_SCORE_HSVAR] = (np.mean([O.rolling_band_mean(g, z_window) for g in self.g_a], axis=0)
                                                    - np.mean([O.rolling_band_mean(g, z_window) for g in self.g_b], axis=0))
        if kinds & KV_KINDS:
            for kind, u in kv_u_traces(model, tabs, seq, length, kinds, lag).items():
                self.scores[kind] = O.rolling_mean(u, lag_window)


def _trace_check(self, kind, pos, gpu, what=""):
    """GPU scores of `kind` at positions `pos` against this trace's oracle."""
    cond = self.cond.get(kind)
    assert_scores_close(gpu, self.scores[kind][pos], what, None if cond is None else cond[pos])


OracleTrace.check = _trace_check


class Session:
    """One context + K/V pool driven call by call from the host."""

    def __init__(self, model, *, n_seq, kinds, layout, max_tokens, max_new, prefill, policies,
                 z_window=64, lag=16, lag_window=64, recency_cap=128, block_size=16, shuffle_blocks=True,
                 select_chunk=1, layer_budgets=0, layer_tables=False, device="cuda"):
        self.m = model
        self.n_seq = n_seq
        self.kinds = kinds
        self.prefill = list(prefill)
        self.policies = list(policies)
        self.recency_cap = recency_cap
        self.select_chunk = select_chunk
        self.layer_budgets = layer_budgets
        self.L = model.num_layers
        self.max_new = max_new
        self.dt = DeviceTrace(model, device)
        self.cfg = E.make_config(max_seqs=n_seq, max_cache_tokens=max_tokens, max_new_tokens=max_new,
                                 num_layers=model.num_layers, num_kv_heads=model.num_kv_heads,
                                 head_dim=model.head_dim, hidden=model.hidden, n_band_a=len(model.band_a),
                                 n_band_b=len(model.band_b), z_window=z_window, lag=lag, lag_window=lag_window,
                                 recency_cap=recency_cap, score_kinds=kinds, select_chunk=select_chunk,
                                 layer_budgets=layer_budgets)
        nbytes = E.epikv_workspace_bytes(self.cfg)
        assert nbytes > 0
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.ctx = E.epikv_init(self.cfg, self.ws, nbytes)
        for b in range(n_seq):
            E.epikv_seq_reset(self.ctx, b, self.prefill[b], self.policies[b])
        bt = None
        self.layer_tables = layer_tables and layout == E.EPIKV_LAYOUT_PAGED
        if layout == E.EPIKV_LAYOUT_PAGED:
            mb = (max_tokens + block_size - 1) // block_size
            nt = n_seq * mb * (model.num_layers if self.layer_tables else 1)
            perm = gen.block_permutation(model.seed, nt) if shuffle_blocks else np.arange(nt)
            bt = perm.reshape(model.num_layers, n_seq, mb) if self.layer_tables else perm.reshape(n_seq, mb)
        self.cache = KVCache(layout, model.num_layers, model.num_kv_heads, model.head_dim, max_seqs=n_seq,
                             max_tokens=max_tokens, block_size=block_size, block_table=bt,
                             layer_tables=self.layer_tables, device=device)
        self.bt_host = None if bt is None else np.asarray(bt)
        # canary fill: any row the library wrongly writes or reads stands out
        self.cache.k.view(torch.int16).fill_(0x7FC1)
        self.cache.v.view(torch.int16).fill_(0x7FC2)
        self.kv = self.cache.view()
        nb = len(model.band_a) + len(model.band_b)
        self.hid = torch.empty((nb, n_seq * max_new, model.hidden), dtype=torch.bfloat16, device=device) \
            if kinds & BAND_KINDS else None
        self.n_cache = [0] * n_seq
        self.n_seen = [0] * n_seq
        lay = (self.L,) if layer_budgets else ()
        self.kept = torch.empty((n_seq,) + lay + (max_tokens,), dtype=torch.int32, device=device)
        self.n_kept = torch.empty((n_seq,) + lay, dtype=torch.int32, device=device)
        # per-layer budgets: each layer's length, and a one-sequence staging
        # cache the new rows are generated into before each layer's copy
        self.n_layer = [[0] * self.L for _ in range(n_seq)]
        self.stage = KVCache(E.EPIKV_LAYOUT_CONTIGUOUS, model.num_layers, model.num_kv_heads, model.head_dim,
                             max_seqs=1, max_tokens=max_new, device=device) \
            if layer_budgets or self.layer_tables else None

    # ---------------------------------------------------------------- inputs
    def append(self, entries):
        """Generate the new tokens' K/V into the cache and their band rows into
        the packed staging buffer; return (seq_ids, cu_new, max_new, hidden view)."""
        cu = [0]
        for b, n in entries:
            assert self.n_cache[b] + n <= self.cache.T
            if self.stage is not None:   # per-layer slots or per-layer block tables: layer by layer
                kw = self.stage.synth_kwargs()
                kw["stride_seq"] = 0
                self.dt.kv(b, self.n_seen[b], n, 0, self.stage.k, self.stage.v, **kw)
                for l in range(self.L):
                    first = self.n_layer[b][l] if self.layer_budgets else self.n_cache[b]
                    slots = np.arange(first, first + n)
                    for kind, pool in ((0, self.stage.k), (1, self.stage.v)):
                        self.cache.write_layer_rows(kind, b, l, slots, pool[l, 0, :n], self.bt_host)
            else:
                self.dt.kv(b, self.n_seen[b], n, self.n_cache[b], self.cache.k, self.cache.v,
                           **self.cache.synth_kwargs())
            if self.hid is not None:
                for i, layer in enumerate(self.m.band_layers):
                    out = self.hid[i, cu[-1]:cu[-1] + n]
                    self.dt.hidden(b, layer, self.n_seen[b], n, out, self.m.hidden)
            cu.append(cu[-1] + n)
        seq_ids = torch.tensor([b for b, _ in entries], dtype=torch.int32, device=self.ws.device)
        cu_new = torch.tensor(cu, dtype=torch.int32, device=self.ws.device)
        hv = None
        if self.hid is not None:
            hv = E.hidden_view([self.hid[i] for i in range(self.hid.shape[0])], self.m.hidden)
        mx = max([n for _, n in entries] + [0])
        return seq_ids, cu_new, mx, hv

    def score_update(self, entries):
        seq_ids, cu_new, mx, hv = self.append(entries)
        E.epikv_score_update(self.ctx, len(entries), seq_ids, cu_new, mx, hv, self.kv)
        for b, n in entries:
            self.n_cache[b] += n
            self.n_seen[b] += n
            self.n_layer[b] = [x + n for x in self.n_layer[b]]
        self._keep_alive = (seq_ids, cu_new)

    def step(self, entries, budgets, triggers):
        """One epikv_step (score + device trigger + select + compact)."""
        seq_ids, cu_new, mx, hv = self.append(entries)
        n = len(entries)
        bud = torch.tensor(budgets, dtype=torch.int32, device=self.ws.device)
        trig = torch.tensor(triggers, dtype=torch.int32, device=self.ws.device)
        out = torch.empty((n, self.L) if self.layer_budgets else (n,), dtype=torch.int32, device=self.ws.device)
        E.epikv_step(self.ctx, n, seq_ids, cu_new, mx, bud, trig, hv, self.kv, out)
        lens = out.cpu().numpy()
        for i, (b, k) in enumerate(entries):
            self.n_seen[b] += k
            if self.layer_budgets:
                self.n_layer[b] = [int(x) for x in lens[i]]
                self.n_cache[b] = max(self.n_layer[b])
            else:
                self.n_cache[b] = int(lens[i])

    def read(self, b, kind):
        pos, sc, n = E.epikv_read_slots(self.ctx, b, kind, self.cache.T)
        assert n == self.n_cache[b], (n, self.n_cache[b])
        return np.array(pos, dtype=np.int64), np.array(sc, dtype=np.float32)

    def select(self, seqs, budgets, triggers=None):
        seq_ids = torch.tensor(seqs, dtype=torch.int32, device=self.ws.device)
        bud = torch.tensor(budgets, dtype=torch.int32, device=self.ws.device)
        trig = None if triggers is None else torch.tensor(triggers, dtype=torch.int32, device=self.ws.device)
        E.epikv_select(self.ctx, len(seqs), seq_ids, bud, trig, self.kept, self.kept.shape[-1], self.n_kept)
        torch.cuda.synchronize()
        nk = self.n_kept[:len(seqs)].cpu().numpy()
        kept = self.kept[:len(seqs)].cpu().numpy()
        self._sel = (seq_ids,)
        out = {}
        if self.layer_budgets:   # {b: per-layer kept lists} of the entries where some layer evicted
            for i, b in enumerate(seqs):
                if any(nk[i, l] < self.n_layer[b][l] for l in range(self.L)):
                    out[b] = [kept[i, l, :nk[i, l]].astype(np.int64) for l in range(self.L)]
                self.n_layer[b] = [int(x) for x in nk[i]]
                self.n_cache[b] = max(self.n_layer[b])
            return out
        for i, b in enumerate(seqs):
            if nk[i] < self.n_cache[b]:
                out[b] = kept[i, :nk[i]].astype(np.int64)
            self.n_cache[b] = int(nk[i])
        return out

    def compact(self, seqs):
        seq_ids = torch.tensor(seqs, dtype=torch.int32, device=self.ws.device)
        E.epikv_compact(self.ctx, len(seqs), seq_ids, self.kept, self.kept.shape[-1], self.kv)
        self._cmp = seq_ids

    def read_layer(self, b, layer):
        pos, n = E.epikv_read_layer_slots(self.ctx, b, layer, self.cache.T)
        assert n == self.n_layer[b][layer], (b, layer, n, self.n_layer[b][layer])
        return np.array(pos, dtype=np.int64)

    def layer_rows_u16(self, b, layer, slots):
        k = as_u16(self.cache.rows(0, b, slots, self.bt_host)[:, layer])
        v = as_u16(self.cache.rows(1, b, slots, self.bt_host)[:, layer])
        return k, v

    def error(self):
        return E.epikv_get_error(self.ctx)

    def cache_rows_u16(self, b, slots):
        k = as_u16(self.cache.rows(0, b, slots, self.bt_host))
        v = as_u16(self.cache.rows(1, b, slots, self.bt_host))
        return k, v

    def close(self):
        E.epikv_destroy(self.ctx)


def kernel_chunk_mean(values):
    """A chunk's mean as the selection kernel forms it from fp32 scores: the
    members summed left to right in fp32, divided by the count in fp32.  The
    exact replay of the GPU's selection on its own scores ranks chunks by this
    value (the oracle's R18 mean is fp64); the fp64 check of the same kept set
    then allows the difference near the threshold."""
    s = np.float32(0.0)
    for v in values:
        s = np.float32(s + np.float32(v))
    return float(np.float32(s / np.float32(len(values))))


def oracle_kept(sc, pos, K, P, cap, chunk=1):
    """The oracle's selection replayed on the GPU's own fp32 scores:
    token-level, or chunk-level (with the kernel's fp32 chunk mean) for
    chunk > 1."""
    if chunk > 1:
        return O.select_kept_chunked(np.asarray(sc, np.float64), pos, K, P, cap, chunk, mean=kernel_chunk_mean)
    return O.select_kept(np.asarray(sc, np.float64), K, P, cap)


class LayerReplay:
    """The oracle's per-layer caches of one sequence, replayed on the GPU's
    frozen scores with the same schedule."""

    def __init__(self, n_layers, budgets, prefill, trigger):
        self.caches = [[] for _ in range(n_layers)]
        self.budgets, self.prefill, self.trigger = list(budgets), prefill, trigger
        self.score = {}

    def append(self, positions, scores):
        for p, s in zip(positions, scores):
            self.score[int(p)] = float(s)
        for c in self.caches:
            c.extend(int(p) for p in positions)

    def event(self, recency_cap=128):
        n = max(len(c) for c in self.caches)
        if not (n > self.trigger and n > min(self.budgets)):
            return False
        R = O.layer_recency(self.budgets, self.prefill, n, recency_cap)
        self.caches = [[c[i] for i in O.select_kept_layer([self.score[p] for p in c], K, self.prefill, R)]
                       for c, K in zip(self.caches, self.budgets)]
        return True


def check_selection(kept_gpu, pos_pre, sc_gpu_pre, sc_ref_pre, K, P, cap, chunk=1, cond_pre=None):
    """Exact check on the GPU's own scores + threshold-tie check on fp64
    (cond_pre: the scores' condition numbers, see score_bound)."""
    exp = oracle_kept(sc_gpu_pre, pos_pre, K, P, cap, chunk)
    assert list(kept_gpu) == exp, "selection differs from the oracle run on the GPU's scores"
    if chunk > 1:
        _check_chunk_ties(kept_gpu, pos_pre, sc_ref_pre, K, P, cap, chunk, cond_pre)
        return
    ref = O.select_kept(sc_ref_pre, K, P, cap)
    if list(kept_gpu) != ref:
        n = len(sc_ref_pre)
        Pp = min(P, n)
        R = min(min(cap, K // 4), max(0, K - Pp))
        M = max(0, K - Pp - R)
        cand = sorted(range(Pp, n - R), key=lambda i: (np.isnan(sc_ref_pre[i]), -sc_ref_pre[i], i))
        theta = sc_ref_pre[cand[M - 1]] if M > 0 else np.inf
        c_th = 0.0 if cond_pre is None or M == 0 else cond_pre[cand[M - 1]]
        diff = set(kept_gpu) ^ set(ref)
        for i in diff:
            c_i = 0.0 if cond_pre is None else cond_pre[i]
            allowed = max(TOL * max(1.0, abs(theta)), 2.0 * U32 * (c_i + c_th))
            assert abs(sc_ref_pre[i] - theta) <= allowed, \
                f"slot {i} differs from the fp64 selection away from the threshold"


def _check_chunk_ties(kept_gpu, pos_pre, sc_ref_pre, K, P, cap, chunk, cond_pre=None):
    """Against fp64 scores, chunk-level: a slot may differ only if its chunk's
    mean is within the tolerance of the boundary chunk's mean."""
    ref = O.select_kept_chunked(sc_ref_pre, pos_pre, K, P, cap, chunk)
    diff = set(kept_gpu) ^ set(ref)
    if not diff:
        return
    n = len(sc_ref_pre)
    Pp = min(P, n)
    R = min(min(cap, K // 4), max(0, K - Pp))
    M = max(0, K - Pp - R)
    chunks = O.chunk_scores(sc_ref_pre, pos_pre, range(Pp, n - R), chunk)
    mean_of = {i: float(m) for m, slots in chunks.values() for i in slots}
    order = sorted(chunks, key=lambda c: (np.isnan(chunks[c][0]), -chunks[c][0], c))
    filled, theta = 0, np.inf
    for c in order:
        filled += len(chunks[c][1])
        if filled >= M:
            theta = float(chunks[c][0])
            break
    c_max = 0.0 if cond_pre is None else float(np.max(np.asarray(cond_pre)[list(range(Pp, n - R))], initial=0.0))
    for i in diff:
        allowed = max(TOL * max(1.0, abs(theta)), 4.0 * U32 * c_max)
        assert abs(mean_of[i] - theta) <= allowed, \
            f"slot {i} differs from the fp64 chunk selection away from the threshold"


def oracle_bandz_at(model, tabs, seq, t, w=64):
    """fp64 EpiKV score of position t from the generator's rows of its window."""
    if t == 0:
        return 0.0
    lo = max(0, t - w)
    pos = np.arange(lo, t + 1)
    seg = gen.segment_index(model, seq, t + 1)
    z = {}
    for l in model.band_layers:
        rows = gen.bf16_bits_to_f64(host.hidden_rows(model, tabs, seq, l, pos, seg))
        g = [O.hidden_change(rows[i - 1], rows[i]) for i in range(1, len(pos))]   # positions lo+1 .. t
        window = g[-min(w, t):]
        z[l] = [O.window_zscore(window)]
    return float(O.epiphany_score([z[l] for l in model.band_a], [z[l] for l in model.band_b])[0])


def oracle_hsvar_at(model, tabs, seq, t, w=64):
    """fp64 HS-variance score of position t from the rows of its window."""
    if t == 0:
        return 0.0
    lo = max(0, t - w)
    pos = np.arange(lo, t + 1)
    seg = gen.segment_index(model, seq, t + 1)
    m = {}
    for l in model.band_layers:
        rows = gen.bf16_bits_to_f64(host.hidden_rows(model, tabs, seq, l, pos, seg))
        # g[0] stands for position lo (never inside the window), g[j] for lo + j
        g = np.array([np.nan] + [O.hidden_change(rows[i - 1], rows[i]) for i in range(1, len(pos))])
        m[l] = O.rolling_band_mean(g, w)[-1]
    return float(np.mean([m[l] for l in model.band_a]) - np.mean([m[l] for l in model.band_b]))


def oracle_kv_at(model, tabs, seq, t, kind, w=64):
    """fp64 KV-key / KV-val score of position t."""
    pos = np.arange(max(0, t - w + 1), t + 1)
    sp = gen.spike_flags(model, seq, t + 1)
    X = gen.bf16_bits_to_f64(host.kv_rows(model, tabs, seq, 0 if kind == E.EPIKV_SCORE_KVKEY else 1, pos, sp))
    return float(O.rolling_mean(np.array([O.head_variance(X[i]) for i in range(len(pos))]), w)[-1])


def oracle_score_at(model, tabs, seq, t, kind):
    if kind == E.EPIKV_SCORE_BANDZ:
        return oracle_bandz_at(model, tabs, seq, t)
    if kind == E.EPIKV_SCORE_HSVAR:
        return oracle_hsvar_at(model, tabs, seq, t)
    if kind in (E.EPIKV_SCORE_KVKEY, E.EPIKV_SCORE_KVVAL):
        return oracle_kv_at(model, tabs, seq, t, kind)
    return oracle_lag_at(model, tabs, seq, t, key_only=kind == E.EPIKV_SCORE_LAGKEY)


def oracle_lag_at(model, tabs, seq, t, lag=16, w=64, key_only=False):
    """fp64 Lag-KV score of position t from the generator's rows it depends on."""
    t0 = max(0, t - w + 1)
    first = max(0, (t0 // lag - 1) * lag)
    pos = np.arange(first, t + 1)
    sp = gen.spike_flags(model, seq, t + 1)
    K = gen.bf16_bits_to_f64(host.kv_rows(model, tabs, seq, 0, pos, sp))
    V = gen.bf16_bits_to_f64(host.kv_rows(model, tabs, seq, 1, pos, sp))
    u = []
    for tt in range(t0, t + 1):
        c = tt // lag
        if c == 0:
            u.append(0.0)
        elif key_only:
            lo = (c - 1) * lag - first
            u.append(O.lag_key_token_variance(K[tt - first], K[lo:lo + lag]))
        else:
            lo = (c - 1) * lag - first
            u.append(O.lag_token_variance(K[tt - first], V[tt - first], K[lo:lo + lag], V[lo:lo + lag]))
    return float(O.rolling_mean(np.array(u), w)[-1])


def check_compaction_sampled(sess, b, pos_after, n_rows, rng):
    """Compacted rows at `n_rows` random slots (every layer, head, K and V)."""
    slots = np.sort(rng.choice(len(pos_after), size=min(n_rows, len(pos_after)), replace=False))
    sp = gen.spike_flags(sess.m, b, int(pos_after.max()) + 1)
    k, v = sess.cache_rows_u16(b, slots)
    np.testing.assert_array_equal(k, host.kv_rows(sess.m, sess.dt.tabs, b, 0, pos_after[slots], sp))
    np.testing.assert_array_equal(v, host.kv_rows(sess.m, sess.dt.tabs, b, 1, pos_after[slots], sp))


def check_compaction(sess, b, pos_after):
    """Compacted rows of every layer and head equal the generator's rows."""
    sp = gen.spike_flags(sess.m, b, int(pos_after.max()) + 1)
    tabs = sess.dt.tabs
    k, v = sess.cache_rows_u16(b, np.arange(len(pos_after)))
    np.testing.assert_array_equal(k, host.kv_rows(sess.m, tabs, b, 0, pos_after, sp))
    np.testing.assert_array_equal(v, host.kv_rows(sess.m, tabs, b, 1, pos_after, sp))
