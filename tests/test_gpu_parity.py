"""GPU parity of the CUDA path against the fp64 oracle, through the C ABI, at
sizes the oracle finishes in seconds (several tiles, ragged tails)."""
import numpy as np
import pytest
import torch

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from synth import gen, workloads as W
from synth.device import DeviceTrace, as_u16

from .harness import ALL_KINDS, OracleTrace, Session, check_compaction, check_selection

pytestmark = pytest.mark.gpu


def test_generator_device_twin_is_bit_identical(gpu_lib):
    for model in (W.small_model(11), gen.TraceModel(0xE91C0002)):
        dt = DeviceTrace(model)
        T = 300
        seg = gen.segment_index(model, 3, T)
        out = torch.empty((T, model.hidden), dtype=torch.bfloat16, device="cuda")
        for layer in (model.band_a[0], model.band_b[-1]):
            dt.hidden(3, layer, 0, T, out, model.hidden)
            np.testing.assert_array_equal(as_u16(out), gen.hidden_rows(model, dt.tabs, 3, layer, np.arange(T), seg))
        from paper_2606_26472_gb300.cache import KVCache
        for layout in (E.EPIKV_LAYOUT_CONTIGUOUS, E.EPIKV_LAYOUT_PAGED):
            bt = gen.block_permutation(5, 4 * 20).reshape(4, 20) if layout else None
            c = KVCache(layout, model.num_layers, model.num_kv_heads, model.head_dim, max_seqs=4, max_tokens=320,
                        block_table=bt)
            dt.kv(2, 1000, 150, 7, c.k, c.v, **c.synth_kwargs())
            sp = gen.spike_flags(model, 2, 1150)
            slots = np.arange(7, 157)
            np.testing.assert_array_equal(as_u16(c.rows(0, 2, slots, bt)),
                                          gen.kv_rows(model, dt.tabs, 2, 0, np.arange(1000, 1150), sp))
            np.testing.assert_array_equal(as_u16(c.rows(1, 2, slots, bt)),
                                          gen.kv_rows(model, dt.tabs, 2, 1, np.arange(1000, 1150), sp))


CASES = [
    # layout, kinds, prefill, budgets, new-token pattern, lag, selection chunk C
    ("contig_bandz", E.EPIKV_LAYOUT_CONTIGUOUS, E.EPIKV_SCORE_BANDZ, (0, 5, 0), (100, 60, 130), (7, 1, 33), 16, 1),
    ("paged_lag", E.EPIKV_LAYOUT_PAGED, E.EPIKV_SCORE_LAGKV, (0, 0, 20), (100, 64, 90), (16, 5, 40), 16, 1),
    ("paged_both", E.EPIKV_LAYOUT_PAGED, E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV, (3, 0, 0), (80, 120, 50),
     (1, 9, 64), 5, 1),
    ("contig_all_kinds_a", E.EPIKV_LAYOUT_CONTIGUOUS, 63, (0, 2, 0), (90, 70, 110), (5, 16, 23), 16, 1),
    ("paged_all_kinds_b", E.EPIKV_LAYOUT_PAGED, 63, (0, 0, 9), (60, 100, 75), (32, 3, 12), 7, 1),
    # long prefixes: P = 100 < K, P = 1, and P = 100 > K (the whole prefill kept, no recency window)
    ("contig_bandz_prefill100", E.EPIKV_LAYOUT_CONTIGUOUS, E.EPIKV_SCORE_BANDZ, (100, 1, 100), (150, 64, 64),
     (7, 1, 33), 16, 1),
    # chunk-level selection
    ("contig_bandz_chunk4", E.EPIKV_LAYOUT_CONTIGUOUS, E.EPIKV_SCORE_BANDZ, (0, 5, 0), (100, 60, 130), (7, 1, 33),
     16, 4),
    ("paged_lag_chunk16", E.EPIKV_LAYOUT_PAGED, E.EPIKV_SCORE_LAGKV, (0, 0, 20), (100, 64, 90), (16, 5, 40), 16,
     16),
    ("paged_both_chunk3", E.EPIKV_LAYOUT_PAGED, E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV, (3, 0, 0),
     (80, 120, 50), (1, 9, 64), 5, 3),
]

# the policy driving each of the three sequences' selection, per case
POLICIES = {
    "contig_all_kinds_a": (E.EPIKV_SCORE_HSVAR, E.EPIKV_SCORE_KVKEY, E.EPIKV_SCORE_LAGKEY),
    "paged_all_kinds_b": (E.EPIKV_SCORE_KVVAL, E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV),
}


@pytest.mark.parametrize("name,layout,kinds,prefill,budgets,chunks,lag,select_chunk", CASES,
                         ids=[c[0] for c in CASES])
def test_decode_parity_small(gpu_lib, name, layout, kinds, prefill, budgets, chunks, lag, select_chunk):
    model = W.small_model(1000 + len(name))
    n_seq = 3
    lengths = (310, 257, 333)
    slack = 12
    policies = list(POLICIES.get(name) or
                    [E.EPIKV_SCORE_BANDZ if (kinds & 1 and (b % 2 == 0 or kinds == 1)) else E.EPIKV_SCORE_LAGKV
                     for b in range(n_seq)])
    max_new = max(chunks)
    T_cap = max(budgets) + slack + max_new + 1
    sess = Session(model, n_seq=n_seq, kinds=kinds, layout=layout, max_tokens=T_cap, max_new=max_new,
                   prefill=prefill, policies=policies, lag=lag, select_chunk=select_chunk)
    refs = [OracleTrace(model, sess.dt.tabs, b, lengths[b], kinds, lag=lag) for b in range(n_seq)]
    events = 0
    step = 0
    while any(sess.n_seen[b] < lengths[b] for b in range(n_seq)):
        entries = []
        for b in range(n_seq):
            n = min(chunks[(b + step) % len(chunks)], lengths[b] - sess.n_seen[b])
            if n > 0:
                entries.append((b, n))
        step += 1
        before = {b: sess.n_cache[b] for b, _ in entries}
        sess.score_update(entries)
        pre = {}
        for b, n in entries:
            for kind in ALL_KINDS:
                if kinds & kind:
                    pos, sc = sess.read(b, kind)
                    new = slice(before[b], before[b] + n)
                    np.testing.assert_array_equal(pos[new], np.arange(sess.n_seen[b] - n, sess.n_seen[b]))
                    refs[b].check(kind, pos[new], sc[new], f"{name} seq {b} kind {kind}")
                    if kind == policies[b]:
                        pre[b] = (pos, sc)
        seqs = [b for b, _ in entries]
        kept = sess.select(seqs, [budgets[b] for b in seqs], [budgets[b] + slack for b in seqs])
        sess.compact(seqs)
        for b, kl in kept.items():
            events += 1
            pos, sc = pre[b]
            cond = refs[b].cond.get(policies[b])
            check_selection(kl, pos, sc, refs[b].scores[policies[b]][pos], budgets[b], prefill[b], 128,
                            select_chunk, None if cond is None else cond[pos])
            pos_after, _ = sess.read(b, policies[b])
            np.testing.assert_array_equal(pos_after, pos[kl])
            check_compaction(sess, b, pos_after)
    assert events >= 6
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


@pytest.mark.parametrize("kinds", [63, E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_HSVAR, 58],
                         ids=["all_kinds", "band_kinds", "kv_kinds"])
def test_chunking_invariance_and_causality(gpu_lib, kinds):
    """Scores are identical, bit for bit, however the trace is split into calls
    (one token per call takes the one-launch decode kernels -- band kinds
    alone the fused g + z kernel, with a K/V kind the kernel that also runs
    the K/V streams -- and the longer calls the multi-kernel path)."""
    model = W.small_model(77)
    L = 200
    results = []
    for chunk in (1, 7, 64, 200):
        sess = Session(model, n_seq=1, kinds=kinds, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=L,
                       max_new=chunk, prefill=(0,), policies=(kinds & -kinds,))
        while sess.n_seen[0] < L:
            sess.score_update([(0, min(chunk, L - sess.n_seen[0]))])
        results.append([sess.read(0, k)[1] for k in ALL_KINDS if kinds & k])
        sess.close()
    for r in results[1:]:
        for a, b in zip(r, results[0]):
            np.testing.assert_array_equal(a, b)


def test_constant_signal_gives_exact_zero_and_lowest_slot_ties(gpu_lib):
    """Hidden rows on a constant-step walk: g is constant, z is exactly 0, so
    every score ties and the kept candidates are the lowest slots."""
    model = W.small_model(5)
    T, K = 240, 100
    sess = Session(model, n_seq=1, kinds=E.EPIKV_SCORE_BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=T,
                   max_new=T, prefill=(0,), policies=(1,))
    rows = torch.zeros((3, T, model.hidden), dtype=torch.bfloat16, device="cuda")
    rows[:, :, 0] = torch.arange(T, device="cuda").remainder(2).to(torch.bfloat16)[None, :]  # 0,1,0,1: |step| 1
    seq_ids = torch.zeros(1, dtype=torch.int32, device="cuda")
    cu = torch.tensor([0, T], dtype=torch.int32, device="cuda")
    hv = E.hidden_view([rows[i] for i in range(3)], model.hidden)
    E.epikv_score_update(sess.ctx, 1, seq_ids, cu, T, hv, sess.kv)
    sess.n_cache[0] = sess.n_seen[0] = T
    pos, sc = sess.read(0, 1)
    assert np.all(sc == 0.0)
    kept = sess.select([0], [K])[0]
    R = 25
    assert list(kept) == list(range(K - R)) + list(range(T - R, T))
    sess.close()
