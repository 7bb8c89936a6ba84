"""Per-layer budgets on the GPU (the per-layer budgets the paper names as
future work, Sec. 5).  The oracle evicts every layer's cache on its own; the
GPU path keeps the union of the layers with a mask per slot and one ranking.
Checked: every layer's positions after every event equal the oracle's
replay on the GPU's own scores, every layer's compacted K/V rows are the
generator's rows of those positions, equal budgets give the token-level
path bit for bit, and the one-call step equals the split calls."""
import numpy as np
import pytest

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from synth import gen, workloads as W
from synth.device import as_u16

from .harness import LayerReplay, OracleTrace, Session, assert_scores_close

pytestmark = pytest.mark.gpu

BANDZ, LAGKV = E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV


def _check_layer_bytes(sess, b, layer, positions):
    slots = np.arange(len(positions))
    k, v = sess.layer_rows_u16(b, layer, slots)
    pos = np.asarray(positions)
    sp = gen.spike_flags(sess.m, b, int(pos.max()) + 1)
    np.testing.assert_array_equal(k, gen.kv_rows(sess.m, sess.dt.tabs, b, 0, pos, sp)[:, layer])
    np.testing.assert_array_equal(v, gen.kv_rows(sess.m, sess.dt.tabs, b, 1, pos, sp)[:, layer])


CASES = [
    # layout, kinds, prefill, per-sequence layer budgets (small model: 4 layers), new-token pattern,
    # one block table per layer (a single block pool, stride_layer = 0)
    ("contig_bandz", E.EPIKV_LAYOUT_CONTIGUOUS, BANDZ, (0, 5, 0),
     ((100, 80, 60, 40), (64, 64, 64, 64), (40, 90, 70, 120)), (7, 1, 33), False),
    ("paged_lag", E.EPIKV_LAYOUT_PAGED, LAGKV, (0, 3, 20),
     ((48, 96, 72, 120), (130, 30, 30, 130), (60, 61, 62, 63)), (16, 5, 40), False),
    ("paged_both", E.EPIKV_LAYOUT_PAGED, BANDZ | LAGKV, (3, 0, 0),
     ((80, 50, 110, 20), (33, 66, 99, 132), (90, 90, 45, 45)), (1, 9, 64), False),
    ("paged_both_layer_tables", E.EPIKV_LAYOUT_PAGED, BANDZ | LAGKV, (0, 4, 0),
     ((120, 90, 60, 30), (50, 100, 50, 100), (77, 66, 55, 44)), (5, 16, 33), True),
]


@pytest.mark.parametrize("name,layout,kinds,prefill,budgets,chunks,layer_tables", CASES, ids=[c[0] for c in CASES])
def test_layer_budget_decode_parity_small(gpu_lib, name, layout, kinds, prefill, budgets, chunks, layer_tables):
    model = W.small_model(2000 + len(name))
    n_seq, L = 3, model.num_layers
    lengths = (301, 260, 333)
    slack = 10
    policies = [BANDZ if (kinds & BANDZ and (b % 2 == 0 or kinds == BANDZ)) else LAGKV for b in range(n_seq)]
    max_new = max(chunks)
    T_cap = max(max(k) for k in budgets) + slack + max_new + 1
    sess = Session(model, n_seq=n_seq, kinds=kinds, layout=layout, max_tokens=T_cap, max_new=max_new,
                   prefill=prefill, policies=policies, layer_budgets=1, layer_tables=layer_tables)
    refs = [OracleTrace(model, sess.dt.tabs, b, lengths[b], kinds) for b in range(n_seq)]
    triggers = [max(budgets[b]) + slack for b in range(n_seq)]
    replay = [LayerReplay(L, budgets[b], prefill[b], triggers[b]) for b in range(n_seq)]
    events, step = 0, 0
    while any(sess.n_seen[b] < lengths[b] for b in range(n_seq)):
        entries = []
        for b in range(n_seq):
            n = min(chunks[(b + step) % len(chunks)], lengths[b] - sess.n_seen[b])
            if n > 0:
                entries.append((b, n))
        step += 1
        before = {b: sess.n_cache[b] for b, _ in entries}
        sess.score_update(entries)
        for b, n in entries:
            pos, sc = sess.read(b, policies[b])
            new = slice(before[b], before[b] + n)
            np.testing.assert_array_equal(pos[new], np.arange(sess.n_seen[b] - n, sess.n_seen[b]))
            assert_scores_close(sc[new], refs[b].scores[policies[b]][pos[new]], f"{name} seq {b}")
            replay[b].append(pos[new], sc[new])
        seqs = [b for b, _ in entries]
        kept = sess.select(seqs, [list(budgets[b]) for b in seqs], [triggers[b] for b in seqs])
        sess.compact(seqs)
        for b in seqs:
            fired = replay[b].event()
            assert (b in kept) <= fired
            events += fired
            for l in range(L):
                got = sess.read_layer(b, l)
                assert list(got) == replay[b].caches[l], f"{name} seq {b} layer {l} step {step}"
            if fired and step % 3 == 0:
                for l in range(L):
                    _check_layer_bytes(sess, b, l, replay[b].caches[l])
    assert events >= 6
    for b in range(n_seq):
        for l in range(L):
            _check_layer_bytes(sess, b, l, replay[b].caches[l])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_equal_layer_budgets_are_the_token_path_bit_for_bit(gpu_lib):
    model = W.small_model(63)
    kw = dict(n_seq=2, kinds=BANDZ | LAGKV, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=180, max_new=20,
              prefill=(3, 0), policies=(BANDZ, LAGKV))
    a, b = Session(model, layer_budgets=1, **kw), Session(model, **kw)
    K, slack = (100, 70), 12
    for step in range(25):
        entries = [(s, (7, 20, 3)[(s + step) % 3]) for s in range(2)]
        a.score_update(entries)
        b.score_update(entries)
        ka = a.select([0, 1], [[K[s]] * model.num_layers for s in range(2)], [K[s] + slack for s in range(2)])
        kb = b.select([0, 1], list(K), [K[s] + slack for s in range(2)])
        a.compact([0, 1])
        b.compact([0, 1])
        assert set(ka) == set(kb)
        for s in ka:
            for l in range(model.num_layers):
                np.testing.assert_array_equal(ka[s][l], kb[s])
        for s in range(2):
            assert a.n_cache[s] == b.n_cache[s] and a.n_layer[s] == [b.n_cache[s]] * model.num_layers
            for kind in (BANDZ, LAGKV):
                pa, sa = a.read(s, kind)
                pb, sb = b.read(s, kind)
                np.testing.assert_array_equal(pa, pb)
                np.testing.assert_array_equal(sa.view(np.uint32), sb.view(np.uint32))
    for s in range(2):
        n = a.n_cache[s]
        np.testing.assert_array_equal(np.stack(a.cache_rows_u16(s, np.arange(n))),
                                      np.stack(b.cache_rows_u16(s, np.arange(n))))
    assert E.epikv_get_stats(a.ctx)["layer_rows_moved"] == E.epikv_get_stats(b.ctx)["layer_rows_moved"] > 0
    assert a.error() == b.error() == (E.EPIKV_OK, 0)
    a.close()
    b.close()


def test_token_budgets_over_per_layer_block_tables_equal_the_shared_table(gpu_lib):
    """One block pool with a block table per layer (stride_layer = 0) holds
    the same rows as the layer-plane layout with one shared table, and the
    scores, selections and compacted rows are the same bit for bit."""
    model = W.small_model(66)
    kw = dict(n_seq=3, kinds=BANDZ | LAGKV, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=150, max_new=24,
              prefill=(0, 2, 0), policies=(BANDZ, LAGKV, LAGKV))
    a, b = Session(model, layer_tables=True, **kw), Session(model, **kw)
    assert a.kv.stride_layer == 0 and a.kv.stride_table_layer > 0
    budgets, triggers = [90, 64, 110], [100, 70, 125]
    for step in range(24):
        entries = [(s, (24, 3, 11)[(s + step) % 3]) for s in range(3)]
        a.step(entries, budgets, triggers)
        b.step(entries, budgets, triggers)
        for s in range(3):
            assert a.n_cache[s] == b.n_cache[s]
            for kind in (BANDZ, LAGKV):
                pa, sa = a.read(s, kind)
                pb, sb = b.read(s, kind)
                np.testing.assert_array_equal(pa, pb)
                np.testing.assert_array_equal(sa.view(np.uint32), sb.view(np.uint32))
    for s in range(3):
        n = a.n_cache[s]
        np.testing.assert_array_equal(np.stack(a.cache_rows_u16(s, np.arange(n))),
                                      np.stack(b.cache_rows_u16(s, np.arange(n))))
    assert E.epikv_get_stats(a.ctx)["evictions"] > 20
    assert a.error() == b.error() == (E.EPIKV_OK, 0)
    a.close()
    b.close()


def test_layer_budget_step_equals_split_calls(gpu_lib):
    model = W.small_model(64)
    kw = dict(n_seq=3, kinds=LAGKV, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=220, max_new=24,
              prefill=(0, 4, 1), policies=(LAGKV,) * 3, layer_budgets=1)
    a, b = Session(model, **kw), Session(model, **kw)
    budgets = [[120, 90, 60, 30], [50, 50, 100, 100], [64, 128, 96, 32]]
    triggers = [max(k) + 9 for k in budgets]
    for step in range(30):
        entries = [(s, (24, 2, 11)[(s + step) % 3]) for s in range(3)]
        a.step(entries, budgets, triggers)
        b.score_update(entries)
        b.select([0, 1, 2], budgets, triggers)
        b.compact([0, 1, 2])
        for s in range(3):
            assert a.n_layer[s] == b.n_layer[s]
            for l in range(model.num_layers):
                np.testing.assert_array_equal(a.read_layer(s, l), b.read_layer(s, l))
    for s in range(3):
        for l in range(model.num_layers):
            n = a.n_layer[s][l]
            np.testing.assert_array_equal(np.stack(a.layer_rows_u16(s, l, np.arange(n))),
                                          np.stack(b.layer_rows_u16(s, l, np.arange(n))))
    assert a.error() == b.error() == (E.EPIKV_OK, 0)
    a.close()
    b.close()


def test_a_bad_layer_budget_is_reported_and_nothing_moves(gpu_lib):
    model = W.small_model(65)
    sess = Session(model, n_seq=1, kinds=BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=80, max_new=80,
                   prefill=(0,), policies=(BANDZ,), layer_budgets=1)
    sess.score_update([(0, 80)])
    before = [sess.read_layer(0, l) for l in range(model.num_layers)]
    assert sess.select([0], [[40, 0, 40, 40]]) == {}
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_BUDGET)
    for l in range(model.num_layers):
        np.testing.assert_array_equal(sess.read_layer(0, l), before[l])
    sess.close()


def test_config2_shape_with_pyramid_layer_budgets(gpu_lib):
    """The 8 x 8,192 band-z workload (32 layers, 64 new tokens per call, the
    trigger K_max + 63) with pyramid per-layer budgets 6,144 .. 2,048 (mean
    4,096): every layer's positions of two sequences equal the oracle's
    replay after the first event, mid-way and at the end; every layer ends at
    its budget; sampled slots of every layer hold the generator's rows."""
    wl = W.config(2)
    m = wl.model
    L = m.num_layers
    budgets = W.pyramid_budgets(wl.budgets[0], L)
    K_max = max(budgets)
    sess = Session(m, n_seq=wl.n_seq, kinds=wl.kinds, layout=wl.layout, max_tokens=K_max + wl.chunk,
                   max_new=wl.chunk, prefill=[0] * wl.n_seq, policies=wl.policies, layer_budgets=1)
    trig = K_max + wl.trigger_slack[0]
    checked = (0, 5)
    replay = {b: LayerReplay(L, budgets, 0, trig) for b in checked}
    n_steps = wl.max_len // wl.chunk
    first = trig // wl.chunk                  # the first step that evicts
    rng = np.random.default_rng(7)
    events = 0
    for st in range(n_steps):
        entries = [(b, wl.chunk) for b in range(wl.n_seq)]
        before = {b: sess.n_cache[b] for b in checked}
        sess.score_update(entries)
        for b in checked:
            pos, sc = sess.read(b, sess.policies[b])
            new = slice(before[b], before[b] + wl.chunk)
            replay[b].append(pos[new], sc[new])
        kept = sess.select(list(range(wl.n_seq)), [list(budgets)] * wl.n_seq, [trig] * wl.n_seq)
        sess.compact(list(range(wl.n_seq)))
        for b in checked:
            events += replay[b].event()
        if st >= first:
            assert len(kept) == wl.n_seq, f"step {st}: every sequence evicts"
        if st in (first, 110, n_steps - 1):
            for b in checked:
                for l in range(L):
                    assert list(sess.read_layer(b, l)) == replay[b].caches[l], f"step {st} seq {b} layer {l}"
    assert events == 2 * (n_steps - first)
    assert all(sess.n_layer[b] == list(budgets) for b in range(wl.n_seq))
    for b in checked:
        slots = np.sort(rng.choice(min(budgets), size=24, replace=False))
        k = as_u16(sess.cache.rows(0, b, slots, sess.bt_host))
        v = as_u16(sess.cache.rows(1, b, slots, sess.bt_host))
        sp = gen.spike_flags(m, b, wl.max_len)
        for l in range(L):
            pos = np.asarray(replay[b].caches[l])[slots]
            np.testing.assert_array_equal(k[:, l], gen.kv_rows(m, sess.dt.tabs, b, 0, pos, sp)[:, l])
            np.testing.assert_array_equal(v[:, l], gen.kv_rows(m, sess.dt.tabs, b, 1, pos, sp)[:, l])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


@pytest.mark.parametrize("kinds,policies", [
    (BANDZ | E.EPIKV_SCORE_HSVAR, (BANDZ, E.EPIKV_SCORE_HSVAR)),
    (BANDZ | LAGKV, (LAGKV, BANDZ)),
    (LAGKV | E.EPIKV_SCORE_KVKEY, (E.EPIKV_SCORE_KVKEY, LAGKV)),
], ids=["band_kinds", "band_and_lagkv", "kv_kinds"])
def test_layer_budgets_one_token_per_call(gpu_lib, kinds, policies):
    """Decode steps take the one-launch score kernels (band kinds alone: the
    fused g + z kernel; with a K/V kind: the kernel that also runs every
    layer's K/V streams), which must also advance every layer's length, put
    each layer's new row in that layer's own next slot and mark the new slot
    in every layer."""
    model = W.small_model(67)
    L = model.num_layers
    budgets = [[60, 40, 50, 30], [45, 45, 20, 70]]
    triggers = [max(k) + 3 for k in budgets]
    sess = Session(model, n_seq=2, kinds=kinds, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=80, max_new=1,
                   prefill=(2, 0), policies=policies, layer_budgets=1, layer_tables=True)
    refs = [OracleTrace(model, sess.dt.tabs, b, 150, kinds) for b in range(2)]
    replay = [LayerReplay(L, budgets[b], sess.prefill[b], triggers[b]) for b in range(2)]
    for step in range(150):
        sess.score_update([(0, 1), (1, 1)])
        for b in range(2):
            pos, sc = sess.read(b, sess.policies[b])
            refs[b].check(sess.policies[b], pos[-1:], sc[-1:], f"seq {b} step {step}")
            replay[b].append(pos[-1:], sc[-1:])
        sess.select([0, 1], budgets, triggers)
        sess.compact([0, 1])
        for b in range(2):
            replay[b].event()
            if step % 10 == 9 or step == 149:
                for l in range(L):
                    assert list(sess.read_layer(b, l)) == replay[b].caches[l], f"step {step} seq {b} layer {l}"
    for b in range(2):
        for l in range(L):
            _check_layer_bytes(sess, b, l, replay[b].caches[l])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_many_sequences_past_the_pair_limit(gpu_lib):
    """72 sequences x 4 layers = 288 (sequence, layer) pairs: more than the
    balanced split takes under per-layer budgets (256), so the copy runs on
    per-stream units from the shared counter; every layer's slots and bytes
    follow the per-layer replay."""
    model = W.small_model(0x1A7E)
    n_seq, L = 72, model.num_layers
    budgets = [[60 + (b % 5) * 8, 40 + (b % 3) * 10, 50, 30 + (b % 7) * 4] for b in range(n_seq)]
    slack = 6
    triggers = [max(k) + slack for k in budgets]
    T_cap = max(triggers) + 20 + 1
    sess = Session(model, n_seq=n_seq, kinds=LAGKV, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=T_cap, max_new=20,
                   prefill=(0,) * n_seq, policies=(LAGKV,) * n_seq, layer_budgets=1, layer_tables=True)
    replay = [LayerReplay(L, budgets[b], 0, triggers[b]) for b in range(n_seq)]
    events = 0
    for step in range(8):
        entries = [(b, 20 if (b + step) % 4 else 7) for b in range(n_seq)]
        before = {b: sess.n_cache[b] for b, _ in entries}
        sess.score_update(entries)
        for b, n in entries:
            pos, sc = sess.read(b, LAGKV)
            replay[b].append(pos[before[b]:before[b] + n], sc[before[b]:before[b] + n])
        seqs = list(range(n_seq))
        sess.select(seqs, budgets, triggers)
        sess.compact(seqs)
        for b in seqs:
            events += replay[b].event()
            for l in range(L):
                assert list(sess.read_layer(b, l)) == replay[b].caches[l], f"seq {b} layer {l} step {step}"
    assert events >= 100
    for b in (0, 17, 41, 71):
        for l in range(L):
            _check_layer_bytes(sess, b, l, replay[b].caches[l])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
