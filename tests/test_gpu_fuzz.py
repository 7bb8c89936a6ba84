"""Seeded randomised decodes through the C ABI, each drawing its own model
shape (layers, heads, head size, hidden size, band layers), layout and block
size, score kinds and selection policies, windows, lag, recency cap,
prefill, budgets, trigger, new-token pattern, skipped sequences, batch
order, skipped selections, chunk-level selection and per-layer budgets (with
per-layer block tables), checked against the fp64 oracle: scores within
tolerance, kept lists (or per-layer caches) equal to the oracle's on the
GPU's own scores, compacted rows equal to the generator's.  Some trials also
drive a second context through epikv_step in lockstep and compare the two
bit for bit."""
import numpy as np
import pytest

from paper_2606_26472_gb300 import epikv as E
from synth import gen

from .harness import ALL_KINDS, LayerReplay, OracleTrace, Session, check_compaction, check_selection

pytestmark = pytest.mark.gpu


def _draw(seed):
    rng = np.random.default_rng(seed)
    L = int(rng.integers(3, 6))
    H = int(rng.choice([1, 2, 4]))
    d = int(rng.choice([8, 16, 32, 64]))
    hidden = int(rng.choice([64, 256, 520]))
    order = [int(x) for x in rng.permutation(L)]
    na = int(rng.integers(1, L))
    nbb = int(rng.integers(1, L - na + 1))
    model = gen.TraceModel(0xF0220000 + seed, num_layers=L, hidden=hidden, num_kv_heads=H, head_dim=d,
                           band_a=tuple(sorted(order[:na])), band_b=tuple(sorted(order[na:na + nbb])))
    kinds = int(rng.integers(1, 64))
    enabled = [k for k in ALL_KINDS if kinds & k]
    n_seq = int(rng.integers(1, 4))
    p = dict(
        model=model, kinds=kinds, n_seq=n_seq,
        policies=[int(rng.choice(enabled)) for _ in range(n_seq)],
        layout=int(rng.integers(0, 2)), block_size=int(rng.choice([1, 4, 16])),
        z_window=int(rng.choice([1, 5, 64])), lag=int(rng.choice([1, 3, 16])),
        lag_window=int(rng.choice([1, 7, 64])), cap=int(rng.choice([0, 4, 128])),
        prefill=[int(rng.integers(0, 12)) for _ in range(n_seq)],
        layer_budgets=bool(rng.integers(0, 4) == 0),
        slack=int(rng.integers(0, 12)), use_trigger=bool(rng.integers(0, 4) != 0),
        chunks=tuple(int(x) for x in rng.integers(1, 20, size=3)),
        lengths=[int(rng.integers(60, 200)) for _ in range(n_seq)],
    )
    p["layer_tables"] = p["layer_budgets"] and p["layout"] == E.EPIKV_LAYOUT_PAGED and bool(rng.integers(0, 2))
    p["use_step"] = bool(rng.integers(0, 3) == 0)
    p["select_prob"] = 1.0 if p["use_step"] else float(rng.choice([1.0, 0.6]))
    p["skip_prob"] = float(rng.choice([0.0, 0.25]))
    p["shuffle"] = bool(rng.integers(0, 2))
    p["select_chunk"] = 1 if p["layer_budgets"] else int(rng.choice([1, 1, 2, 5]))
    if p["layer_budgets"]:
        p["budgets"] = [[int(x) for x in rng.integers(8, 80, size=L)] for _ in range(n_seq)]
    else:
        p["budgets"] = [int(rng.integers(8, 80)) for _ in range(n_seq)]
    return p


@pytest.mark.parametrize("seed", range(24))
def test_random_decode_against_the_oracle(gpu_lib, seed):
    p = _draw(seed)
    m, n_seq, kinds = p["model"], p["n_seq"], p["kinds"]
    kmax = [max(k) if p["layer_budgets"] else k for k in p["budgets"]]
    max_new = max(p["chunks"])
    T_cap = max(max(kmax) + p["slack"], max(p["prefill"])) + 4 * max_new + 1   # room for skipped selections
    sess = Session(m, n_seq=n_seq, kinds=kinds, layout=p["layout"], max_tokens=T_cap, max_new=max_new,
                   prefill=p["prefill"], policies=p["policies"], z_window=p["z_window"], lag=p["lag"],
                   lag_window=p["lag_window"], recency_cap=p["cap"], block_size=p["block_size"],
                   select_chunk=p["select_chunk"], layer_budgets=int(p["layer_budgets"]),
                   layer_tables=p["layer_tables"])
    twin = Session(m, n_seq=n_seq, kinds=kinds, layout=p["layout"], max_tokens=T_cap, max_new=max_new,
                   prefill=p["prefill"], policies=p["policies"], z_window=p["z_window"], lag=p["lag"],
                   lag_window=p["lag_window"], recency_cap=p["cap"], block_size=p["block_size"],
                   select_chunk=p["select_chunk"], layer_budgets=int(p["layer_budgets"]),
                   layer_tables=p["layer_tables"]) if p["use_step"] else None
    refs = [OracleTrace(m, sess.dt.tabs, b, p["lengths"][b], kinds, z_window=p["z_window"], lag=p["lag"],
                        lag_window=p["lag_window"]) for b in range(n_seq)]
    srng = np.random.default_rng(seed + 1000)
    triggers = [kmax[b] + p["slack"] for b in range(n_seq)]
    replay = [LayerReplay(m.num_layers, p["budgets"][b], p["prefill"][b],
                          triggers[b] if p["use_trigger"] else kmax[b]) for b in range(n_seq)] \
        if p["layer_budgets"] else None
    step = 0
    while any(sess.n_seen[b] < p["lengths"][b] for b in range(n_seq)):
        entries = [(b, min(p["chunks"][(b + step) % 3], p["lengths"][b] - sess.n_seen[b])) for b in range(n_seq)
                   if sess.n_seen[b] < p["lengths"][b]]
        if len(entries) > 1 and p["skip_prob"] > 0:   # some sequences bring nothing this step
            kept_entries = [e for e in entries if srng.random() >= p["skip_prob"]]
            entries = kept_entries or entries[:1]
        if p["shuffle"]:
            entries = [entries[i] for i in srng.permutation(len(entries))]
        step += 1
        before = {b: sess.n_cache[b] for b, _ in entries}
        sess.score_update(entries)
        pre = {}
        for b, n in entries:
            for kind in ALL_KINDS:
                if not kinds & kind:
                    continue
                pos, sc = sess.read(b, kind)
                new = slice(before[b], before[b] + n)
                np.testing.assert_array_equal(pos[new], np.arange(sess.n_seen[b] - n, sess.n_seen[b]))
                refs[b].check(kind, pos[new], sc[new], f"seed {seed} seq {b} kind {kind}")
                if kind == p["policies"][b]:
                    pre[b] = (pos, sc)
                    if replay:
                        replay[b].append(pos[new], sc[new])
        seqs = [b for b, _ in entries]
        trig = [triggers[b] for b in seqs] if p["use_trigger"] else None
        if twin is not None:   # the same step through epikv_step (no trigger = the budget, K_max per layer)
            twin.step(entries, [p["budgets"][b] for b in seqs], trig or [kmax[b] for b in seqs])
        full = any(sess.n_cache[b] + 2 * max_new > T_cap for b in seqs)   # must evict before it overflows
        if not full and srng.random() >= p["select_prob"]:
            continue
        kept = sess.select(seqs, [p["budgets"][b] for b in seqs], trig)
        sess.compact(seqs)
        if twin is not None:
            for b in seqs:
                assert twin.n_cache[b] == sess.n_cache[b], (seed, step, b)
                if p["layer_budgets"]:
                    assert twin.n_layer[b] == sess.n_layer[b], (seed, step, b)
                for kind in ALL_KINDS:
                    if kinds & kind:
                        pa, sa = sess.read(b, kind)
                        pb, sb = twin.read(b, kind)
                        np.testing.assert_array_equal(pa, pb)
                        np.testing.assert_array_equal(sa.view(np.uint32), sb.view(np.uint32))
        for b in seqs:
            if replay:
                replay[b].event(p["cap"])
                for l in range(m.num_layers):
                    assert list(sess.read_layer(b, l)) == replay[b].caches[l], f"seed {seed} seq {b} layer {l}"
            elif b in kept:
                pos, sc = pre[b]
                pol = p["policies"][b]
                cond = refs[b].cond.get(pol)
                check_selection(kept[b], pos, sc, refs[b].scores[pol][pos], p["budgets"][b], p["prefill"][b],
                                p["cap"], p["select_chunk"], None if cond is None else cond[pos])
                pos_after, _ = sess.read(b, p["policies"][b])
                np.testing.assert_array_equal(pos_after, pos[kept[b]])
                check_compaction(sess, b, pos_after)
    if replay:
        for b in range(n_seq):
            for l in range(m.num_layers):
                pos = np.asarray(replay[b].caches[l])
                k, v = sess.layer_rows_u16(b, l, np.arange(len(pos)))
                sp = gen.spike_flags(m, b, int(pos.max()) + 1)
                np.testing.assert_array_equal(k, gen.kv_rows(m, sess.dt.tabs, b, 0, pos, sp)[:, l])
                np.testing.assert_array_equal(v, gen.kv_rows(m, sess.dt.tabs, b, 1, pos, sp)[:, l])
    if twin is not None:
        for b in range(n_seq):
            n = twin.n_cache[b]
            if p["layer_budgets"]:
                for l in range(m.num_layers):
                    nl = twin.n_layer[b][l]
                    np.testing.assert_array_equal(np.stack(twin.layer_rows_u16(b, l, np.arange(nl))),
                                                  np.stack(sess.layer_rows_u16(b, l, np.arange(nl))))
            else:
                np.testing.assert_array_equal(np.stack(twin.cache_rows_u16(b, np.arange(n))),
                                              np.stack(sess.cache_rows_u16(b, np.arange(n))))
        assert twin.error() == (E.EPIKV_OK, 0)
        twin.close()
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
