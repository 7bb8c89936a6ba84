"""GPU parity at the five workloads' full sizes.

Each test runs its workload's whole decode schedule through the C ABI (the
steps through epikv_step, the kernels bench.py times) and checks, against the
fp64 oracle:
* at sampled eviction events: the kept list of every sequence equals the
  oracle's selection re-run on the GPU's own pre-event scores (exact); the
  positions after the event are the kept ones; the compacted K/V of sampled
  slots of sampled sequences equal the generator's rows byte for byte;
* sampled kept tokens' scores equal the oracle's fp64 score of the same
  position (computed one by one from the rows of its window) within
  1e-4 * max(1, |s|);
* at one event of one sequence per workload, the kept list against the fp64
  oracle's scores of every slot of the pre-event cache (threshold ties
  allowed, as check_selection states).
Configuration 1 is small enough for the full oracle: every score, the fp64
kept set and every compacted row are checked.
"""
import numpy as np
import pytest
import torch

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from paper_2606_26472_gb300.cache import KVCache
from synth import gen, workloads as W
from synth.device import DeviceBatchTrace, DeviceTrace, as_u16

from .harness import (ALL_KINDS, OracleTrace, Session, assert_scores_close, check_compaction,
                      check_compaction_sampled, check_selection, oracle_bandz_at, oracle_kept, oracle_lag_at,
                      oracle_score_at)

pytestmark = pytest.mark.gpu


class _CacheProbe:
    """What the sampled byte check needs from a run that has no Session."""

    def __init__(self, m, dt, cache, bt):
        self.m, self.dt, self.cache, self.bt_host = m, dt, cache, bt

    def cache_rows_u16(self, b, slots):
        return (as_u16(self.cache.rows(0, b, slots, self.bt_host)), as_u16(self.cache.rows(1, b, slots, self.bt_host)))


def _event_checks(sess, pre, kept, budgets, rng, sample_bytes, n_rows=192):
    for b, kl in kept.items():
        pos, sc = pre[b]
        exp = oracle_kept(sc, pos, budgets[b], sess.prefill[b], sess.recency_cap, sess.select_chunk)
        assert list(kl) == exp, f"seq {b}: selection differs from the oracle on the GPU's scores"
        pos_after, _ = sess.read(b, sess.policies[b])
        np.testing.assert_array_equal(pos_after, pos[kl])
        if b in sample_bytes:
            check_compaction_sampled(sess, b, pos_after, n_rows, rng)


def _score_samples(sess, seqs, per_seq, rng, kinds):
    for b in seqs:
        for kind in ALL_KINDS:
            if not kinds & kind:
                continue
            pos, sc = sess.read(b, kind)
            idx = rng.choice(len(pos), size=min(per_seq, len(pos)), replace=False)
            for i in idx:
                t = int(pos[i])
                ref = oracle_score_at(sess.m, sess.dt.tabs, b, t, kind)
                assert_scores_close([sc[i]], [ref], f"seq {b} kind {kind} position {t}")


def _fp64_event_check(sess, b, kl, pos, sc, length, wl, select_chunk=1):
    """The kept list of one sequence at one eviction event against the fp64
    oracle: its scores of every pre-event slot from the whole trace up to the
    event (positions < length), then the exact replay on the GPU's scores
    and the threshold-tie check on the fp64 ones (check_selection)."""
    kind = sess.policies[b]
    ref = OracleTrace(sess.m, sess.dt.tabs, b, length, kind, z_window=wl.z_window, lag=wl.lag,
                      lag_window=wl.lag_window)
    cond = ref.cond.get(kind)
    check_selection(kl, pos, sc, ref.scores[kind][pos], wl.budgets[b], sess.prefill[b], sess.recency_cap,
                    select_chunk, None if cond is None else cond[pos])


def _run_chunked(wl, sampled_steps, sample_bytes, score_seqs, per_seq, select_chunk=1, fp64_event=None):
    """fp64_event = (step, sequence): the sampled event whose kept list is
    also checked against the fp64 oracle's scores of the whole pre-event
    cache."""
    m = wl.model
    rng = np.random.default_rng(wl.model.seed)
    K = wl.budgets[0]
    sess = Session(m, n_seq=wl.n_seq, kinds=wl.kinds, layout=wl.layout, max_tokens=K + wl.chunk,
                   max_new=wl.chunk, prefill=[0] * wl.n_seq, policies=wl.policies, select_chunk=select_chunk)
    budgets = list(wl.budgets)
    triggers = [budgets[b] + wl.trigger_slack[b] for b in range(wl.n_seq)]
    n_steps = wl.max_len // wl.chunk
    events = 0
    fp64_done = False
    for st in range(n_steps):
        entries = [(b, wl.chunk) for b in range(wl.n_seq)]
        if st in sampled_steps:
            sess.score_update(entries)
            pre = {b: sess.read(b, sess.policies[b]) for b in range(wl.n_seq)}
            seqs = list(range(wl.n_seq))
            kept = sess.select(seqs, budgets, triggers)
            sess.compact(seqs)
            assert len(kept) == wl.n_seq, f"step {st}: expected every sequence to evict"
            _event_checks(sess, pre, kept, budgets, rng, sample_bytes)
            if fp64_event is not None and fp64_event[0] == st:
                b = fp64_event[1]
                _fp64_event_check(sess, b, kept[b], *pre[b], (st + 1) * wl.chunk, wl, select_chunk)
                fp64_done = True
            events += 1
        else:
            sess.step(entries, budgets, triggers)
    assert events == len(sampled_steps)
    assert fp64_event is None or fp64_done
    assert all(n == K for n in sess.n_cache)
    _score_samples(sess, score_seqs, per_seq, rng, wl.kinds)
    assert sess.error() == (E.EPIKV_OK, 0)
    stats = E.epikv_get_stats(sess.ctx)
    assert stats["tokens_scored"] == wl.n_seq * wl.max_len
    sess.close()


def test_config1_single_2k_full_oracle(gpu_lib):
    wl = W.config(1)
    m = wl.model
    T, K = wl.max_len, wl.budgets[0]
    sess = Session(m, n_seq=1, kinds=wl.kinds, layout=wl.layout, max_tokens=T, max_new=T, prefill=(0,),
                   policies=wl.policies)
    ref = OracleTrace(m, sess.dt.tabs, 0, T, wl.kinds)
    sess.score_update([(0, T)])
    pos, sc = sess.read(0, E.EPIKV_SCORE_BANDZ)
    np.testing.assert_array_equal(pos, np.arange(T))
    assert_scores_close(sc, ref.scores[E.EPIKV_SCORE_BANDZ][pos], "config 1")
    kept = sess.select([0], [K], [K + wl.trigger_slack[0]])
    sess.compact([0])
    check_selection(kept[0], pos, sc, ref.scores[E.EPIKV_SCORE_BANDZ][pos], K, 0, 128)
    pos_after, _ = sess.read(0, E.EPIKV_SCORE_BANDZ)
    np.testing.assert_array_equal(pos_after, pos[kept[0]])
    check_compaction(sess, 0, pos_after)
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_config2_batch8_8k_bandz(gpu_lib):
    wl = W.config(2)
    first = wl.budgets[0] // wl.chunk            # the first step that evicts
    _run_chunked(wl, {first, 100, wl.max_len // wl.chunk - 1}, sample_bytes={0, 5}, score_seqs=range(8),
                 per_seq=6, fp64_event=(100, 3))


def test_config2_shape_with_chunk_level_selection(gpu_lib):
    """The 8 x 8,192 band-z workload with chunk-level selection (16-position
    chunks), every step through epikv_step except the sampled events."""
    wl = W.config(2)
    first = wl.budgets[0] // wl.chunk
    _run_chunked(wl, {first, 77, wl.max_len // wl.chunk - 1}, sample_bytes={3}, score_seqs=(2,), per_seq=3,
                 select_chunk=16, fp64_event=(77, 6))


def test_config2_shape_with_all_six_score_kinds(gpu_lib):
    """The 8 x 8,192 band-z workload's shape with every score kind computed and
    each sequence's selection driven by a different one."""
    import dataclasses
    wl = W.config(2)
    pol = tuple(ALL_KINDS[b % 6] for b in range(wl.n_seq))
    wl = dataclasses.replace(wl, kinds=63, policies=pol)
    first = wl.budgets[0] // wl.chunk
    _run_chunked(wl, {first, wl.max_len // wl.chunk - 1}, sample_bytes={1, 4}, score_seqs=range(6), per_seq=3,
                 fp64_event=(first, 5))


def test_config3_batch32_32k_lagkv_paged(gpu_lib):
    wl = W.config(3)
    first = wl.budgets[0] // wl.chunk
    _run_chunked(wl, {first, 150, wl.max_len // wl.chunk - 1}, sample_bytes={0, 17}, score_seqs=(0, 9, 22, 31),
                 per_seq=4, fp64_event=(150, 22))


def test_config4_batch4_64k_per_token_updates(gpu_lib):
    """65,536 single-token score updates per sequence, then one eviction of
    65,536 -> 4,096 (the radix select runs over 65,408 candidates)."""
    wl = W.config(4)
    m = wl.model
    rng = np.random.default_rng(4)
    Bn, T, K = wl.n_seq, wl.max_len, wl.budgets[0]
    dt = DeviceTrace(m)
    nb = len(m.band_layers)
    hid = torch.empty((nb, T, Bn, m.hidden), dtype=torch.bfloat16, device="cuda")   # [layer][position][seq]
    for i, layer in enumerate(m.band_layers):
        for b in range(Bn):
            dt.hidden(b, layer, 0, T, hid[i, :, b].data_ptr(), Bn * m.hidden)
    cache = KVCache(E.EPIKV_LAYOUT_CONTIGUOUS, m.num_layers, m.num_kv_heads, m.head_dim, max_seqs=Bn, max_tokens=T)
    for b in range(Bn):
        dt.kv(b, 0, T, 0, cache.k, cache.v, **cache.synth_kwargs())
    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=T, max_new_tokens=1, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), score_kinds=E.EPIKV_SCORE_BANDZ)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device="cuda")
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_BANDZ)
    kv = cache.view()
    seq_ids = torch.arange(Bn, dtype=torch.int32, device="cuda")
    cu = torch.arange(Bn + 1, dtype=torch.int32, device="cuda")
    step_bytes = Bn * m.hidden * 2
    bases = [hid[i].data_ptr() for i in range(nb)]
    hv = E.epikv_hidden_view()
    hv.row_stride = m.hidden
    for t in range(T):
        for i in range(nb):
            hv.band_rows[i] = bases[i] + t * step_bytes
        E.epikv_score_update(ctx, Bn, seq_ids, cu, 1, hv, kv)
    del hid
    pre = {}
    for b in range(Bn):
        pos, sc, n = E.epikv_read_slots(ctx, b, E.EPIKV_SCORE_BANDZ, T)
        assert n == T
        pre[b] = (np.array(pos), np.array(sc, dtype=np.float32))
        np.testing.assert_array_equal(pre[b][0], np.arange(T))
    kept = torch.empty((Bn, K), dtype=torch.int32, device="cuda")
    nk = torch.empty(Bn, dtype=torch.int32, device="cuda")
    bud = torch.full((Bn,), K, dtype=torch.int32, device="cuda")
    E.epikv_select(ctx, Bn, seq_ids, bud, None, kept, K, nk)
    E.epikv_compact(ctx, Bn, seq_ids, kept, K, kv)
    torch.cuda.synchronize()
    assert (nk.cpu().numpy() == K).all()
    kept_h = kept.cpu().numpy()

    s = _CacheProbe(m, dt, cache, None)
    # sequence 2's eviction against the fp64 oracle's scores of all 65,536 positions
    ref = OracleTrace(m, dt.tabs, 2, T, E.EPIKV_SCORE_BANDZ)
    check_selection(list(kept_h[2]), pre[2][0], pre[2][1], ref.scores[E.EPIKV_SCORE_BANDZ], K, 0, 128, 1,
                    ref.cond[E.EPIKV_SCORE_BANDZ])
    for b in range(Bn):
        pos, sc = pre[b]
        exp = O.select_kept(sc.astype(np.float64), K, 0, 128)
        assert list(kept_h[b]) == exp
        pos_after, sc_after, n = E.epikv_read_slots(ctx, b, E.EPIKV_SCORE_BANDZ, T)
        assert n == K
        np.testing.assert_array_equal(np.array(pos_after), pos[kept_h[b]])
        check_compaction_sampled(s, b, np.array(pos_after), 192, rng)
        for i in rng.choice(K, size=6, replace=False):
            t = int(pos_after[i])
            assert_scores_close([sc_after[i]], [oracle_bandz_at(m, dt.tabs, b, t)], f"seq {b} position {t}")
    assert E.epikv_get_error(ctx) == (E.EPIKV_OK, 0)
    E.epikv_destroy(ctx)


def test_config5_ragged_continuous_batch_both_scores(gpu_lib):
    """64 sequences of seeded lengths in 4k..32k, one new token per active
    sequence per step, a sequence evicts when its cache exceeds K + 64;
    finished sequences leave the batch."""
    wl = W.config(5)
    m = wl.model
    rng = np.random.default_rng(5)
    Bn = wl.n_seq
    Kmax = max(wl.budgets)
    T_cap = Kmax + wl.trigger_slack[0] + 1
    dt = DeviceBatchTrace(m, Bn, wl.max_len)
    mb = (T_cap + 15) // 16
    bt = gen.block_permutation(m.seed, Bn * mb).reshape(Bn, mb)
    cache = KVCache(E.EPIKV_LAYOUT_PAGED, m.num_layers, m.num_kv_heads, m.head_dim, max_seqs=Bn, max_tokens=T_cap,
                    block_table=bt)
    kv = cache.view()
    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=T_cap, max_new_tokens=1, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), score_kinds=E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device="cuda")
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, wl.policies[b])
    nb = len(m.band_layers)
    hid = torch.empty((nb, Bn, m.hidden), dtype=torch.bfloat16, device="cuda")
    hv = E.hidden_view([hid[i] for i in range(nb)], m.hidden)
    n_cache = [0] * Bn
    lens = np.array(wl.lengths)
    slack = wl.trigger_slack[0]
    n_events = [max(0, (lens[b] - wl.budgets[b] - slack - 1) // (slack + 1) + 1) for b in range(Bn)]
    # the events checked: first, middle and last of the four sequences that evict most
    # (two band-z-policy and two Lag-KV-policy sequences)
    even = sorted(range(0, Bn, 2), key=lambda b: -n_events[b])[:2]
    odd = sorted(range(1, Bn, 2), key=lambda b: -n_events[b])[:2]
    want_events = {b: {0, n_events[b] // 2, n_events[b] - 1} for b in even + odd}
    assert all(n_events[b] >= 3 for b in want_events)
    events_seen = {b: 0 for b in want_events}
    fp64_seqs = {even[1], odd[1]}     # one band-z-policy and one Lag-KV-policy sequence
    fp64_checked = set()
    s = _CacheProbe(m, dt, cache, bt)
    total_events = 0
    out = torch.empty(Bn, dtype=torch.int32, device="cuda")
    for t in range(wl.max_len):
        active = np.nonzero(lens > t)[0]
        n = len(active)
        seqs = torch.from_numpy(active.astype(np.int32)).to("cuda")
        pos = torch.full((n,), t, dtype=torch.int32, device="cuda")
        slots = torch.tensor([n_cache[b] for b in active], dtype=torch.int32, device="cuda")
        dt.kv_batch(seqs, pos, slots, cache.k, cache.v, **cache.synth_kwargs())
        for i, layer in enumerate(m.band_layers):
            dt.hidden_batch(layer, seqs, pos, hid[i], m.hidden)
        cu = torch.arange(n + 1, dtype=torch.int32, device="cuda")
        bud = torch.tensor([wl.budgets[b] for b in active], dtype=torch.int32, device="cuda")
        trig = bud + wl.trigger_slack[0]
        evicting = [b for b in active if n_cache[b] + 1 > wl.budgets[b] + wl.trigger_slack[b]]
        total_events += len(evicting)
        check = [b for b in evicting if b in want_events and events_seen[b] in want_events[b]]
        for b in evicting:
            if b in want_events:
                events_seen[b] += 1
        if check:
            E.epikv_score_update(ctx, n, seqs, cu, 1, hv, kv)
            pre = {}
            for b in check:
                p, sc, nn = E.epikv_read_slots(ctx, b, wl.policies[b], T_cap)
                assert nn == n_cache[b] + 1
                pre[b] = (np.array(p), np.array(sc, dtype=np.float32))
            kept = torch.empty((n, T_cap), dtype=torch.int32, device="cuda")
            E.epikv_select(ctx, n, seqs, bud, trig, kept, T_cap, out)
            E.epikv_compact(ctx, n, seqs, kept, T_cap, kv)
            torch.cuda.synchronize()
            kept_h = kept.cpu().numpy()
            for b in check:
                i = int(np.nonzero(active == b)[0][0])
                K = wl.budgets[b]
                kl = kept_h[i, :K]
                exp = O.select_kept(pre[b][1].astype(np.float64), K, 0, 128)
                assert list(kl) == exp, f"seq {b} event: selection differs from the oracle on the GPU's scores"
                if b in fp64_seqs and events_seen[b] - 1 == n_events[b] // 2:
                    # the middle event against the fp64 oracle's scores of the whole pre-event cache
                    ref = OracleTrace(m, dt.tabs, b, t + 1, wl.policies[b])
                    cond = ref.cond.get(wl.policies[b])
                    pp = pre[b][0]
                    check_selection(list(kl), pp, pre[b][1], ref.scores[wl.policies[b]][pp], K, 0, 128, 1,
                                    None if cond is None else cond[pp])
                    fp64_checked.add(b)
                p_after, _, nn = E.epikv_read_slots(ctx, b, wl.policies[b], T_cap)
                assert nn == K
                np.testing.assert_array_equal(np.array(p_after), pre[b][0][kl])
                check_compaction_sampled(s, b, np.array(p_after), 128, rng)
        else:
            E.epikv_step(ctx, n, seqs, cu, 1, bud, trig, hv, kv, out)
        for b in active:
            n_cache[b] += 1
            if n_cache[b] > wl.budgets[b] + wl.trigger_slack[b]:
                n_cache[b] = wl.budgets[b]
    torch.cuda.synchronize()
    assert total_events > 1000
    assert all(events_seen[b] == n_events[b] for b in want_events)
    assert fp64_checked == fp64_seqs
    for b in range(Bn):
        p, _, nn = E.epikv_read_slots(ctx, b, 1, 1)
        assert nn == n_cache[b], (b, nn, n_cache[b])
    # sampled scores of both kinds, even (band-z policy) and odd (Lag-KV policy) sequences
    for b in (0, 1, 10, 33, 62, 63):
        for kind in (E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV):
            p, sc, nn = E.epikv_read_slots(ctx, b, kind, T_cap)
            for i in rng.choice(nn, size=3, replace=False):
                t = int(p[i])
                ref = oracle_bandz_at(m, dt.tabs, b, t) if kind == 1 else oracle_lag_at(m, dt.tabs, b, t)
                assert_scores_close([sc[i]], [ref], f"seq {b} kind {kind} position {t}")
    assert E.epikv_get_error(ctx) == (E.EPIKV_OK, 0)
    E.epikv_destroy(ctx)
