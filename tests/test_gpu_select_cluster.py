"""The cluster selection (contexts whose caches hold more than 24,576 slots:
one sequence's selection spread over a thread-block cluster of 8 CTAs)
against the one-CTA selection and the oracle.  The same inputs run through a
context with a large capacity (the cluster kernel) and one with a small
capacity (one CTA per sequence); kept lists, scores, positions and compacted
rows must agree bit for bit, and the kept lists equal the oracle's selection
on the GPU's own scores: several evictions, prefill, a recency window that
covers the budget, ties (a constant signal: every score exactly 0), NaN
scores, caches shorter than the cluster and a 30,000-slot cache."""
import numpy as np
import pytest
import torch

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from synth import workloads as W

from .harness import OracleTrace, Session, check_compaction, check_selection

pytestmark = pytest.mark.gpu

BIG = 25000      # capacity above the cluster threshold
KINDS = E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV


def _decode(T_cap, model, lengths, budgets, prefill, chunk, slack):
    n_seq = len(lengths)
    sess = Session(model, n_seq=n_seq, kinds=KINDS, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=T_cap, max_new=chunk,
                   prefill=prefill, policies=[1 + (b % 2) for b in range(n_seq)])
    log = []
    while any(sess.n_seen[b] < lengths[b] for b in range(n_seq)):
        entries = [(b, min(chunk, lengths[b] - sess.n_seen[b])) for b in range(n_seq) if sess.n_seen[b] < lengths[b]]
        sess.score_update(entries)
        seqs = [b for b, _ in entries]
        pre = {b: sess.read(b, sess.policies[b]) for b in seqs}
        kept = sess.select(seqs, [budgets[b] for b in seqs], [budgets[b] + slack for b in seqs])
        sess.compact(seqs)
        for b, kl in kept.items():
            pos, sc = pre[b]
            assert list(kl) == O.select_kept(sc.astype(np.float64), budgets[b], prefill[b], 128)
            log.append((b, list(kl)))
    final = [(sess.read(b, 1), sess.read(b, 2)) for b in range(n_seq)]
    rows = [sess.cache_rows_u16(b, np.arange(sess.n_cache[b])) for b in range(n_seq)]
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
    return log, final, rows


def test_cluster_selection_equals_one_cta_selection_on_decodes(gpu_lib):
    model = W.small_model(91)
    args = dict(lengths=(700, 530, 611), budgets=(200, 96, 300), prefill=(0, 7, 40), chunk=37, slack=20)
    log_c, fin_c, rows_c = _decode(BIG, model, **args)
    log_1, fin_1, rows_1 = _decode(800, model, **args)
    assert len(log_c) >= 20 and log_c == log_1
    for (a, b) in zip(fin_c, fin_1):
        for (p, s), (p1, s1) in zip(a, b):
            np.testing.assert_array_equal(p, p1)
            np.testing.assert_array_equal(s, s1)
    for (k, v), (k1, v1) in zip(rows_c, rows_1):
        np.testing.assert_array_equal(k, k1)
        np.testing.assert_array_equal(v, v1)


@pytest.mark.parametrize("prefill,K", [(30, 20), (20, 24), (0, 1), (5, 6), (0, 3)])
def test_cluster_selection_small_caches_and_budget_edges(gpu_lib, prefill, K):
    """Caches shorter than the cluster (slices of 0 to 7 slots), prefill over
    the budget, recency covering the budget, K = 1."""
    sess = Session(W.small_model(92), n_seq=1, kinds=KINDS, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=BIG,
                   max_new=64, prefill=(prefill,), policies=(1,))
    sess.score_update([(0, 50)])
    pos, sc = sess.read(0, 1)
    kept = sess.select([0], [K])[0]
    assert list(kept) == O.select_kept(sc.astype(np.float64), K, prefill, 128)
    sess.compact([0])
    pos_after, _ = sess.read(0, 1)
    np.testing.assert_array_equal(pos_after, pos[kept])
    check_compaction(sess, 0, pos_after)
    sess.close()


def test_cluster_selection_ties_go_to_the_lowest_slots(gpu_lib):
    """A constant signal: every band-z score is exactly 0, so the kept
    candidates are the lowest slots, across the CTAs of the cluster."""
    model = W.small_model(5)
    T, K = 2400, 1000
    sess = Session(model, n_seq=1, kinds=E.EPIKV_SCORE_BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=BIG,
                   max_new=T, prefill=(0,), policies=(1,))
    rows = torch.zeros((3, T, model.hidden), dtype=torch.bfloat16, device="cuda")
    rows[:, :, 0] = torch.arange(T, device="cuda").remainder(2).to(torch.bfloat16)[None, :]
    seq_ids = torch.zeros(1, dtype=torch.int32, device="cuda")
    cu = torch.tensor([0, T], dtype=torch.int32, device="cuda")
    hv = E.hidden_view([rows[i] for i in range(3)], model.hidden)
    E.epikv_score_update(sess.ctx, 1, seq_ids, cu, T, hv, sess.kv)
    sess.n_cache[0] = sess.n_seen[0] = T
    pos, sc = sess.read(0, 1)
    assert np.all(sc == 0.0)
    kept = sess.select([0], [K])[0]
    R = 128
    assert list(kept) == list(range(K - R)) + list(range(T - R, T))
    sess.close()


def test_cluster_selection_nan_scores_rank_lowest(gpu_lib):
    model = W.small_model(44)
    T, K = 600, 250
    sess = Session(model, n_seq=1, kinds=E.EPIKV_SCORE_BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=BIG,
                   max_new=T, prefill=(0,), policies=(1,))
    seq_ids, cu, mx, hv = sess.append([(0, T)])
    sess.hid[0, 50, 3] = float("nan")
    sess.hid[0, 300, 7] = float("nan")
    E.epikv_score_update(sess.ctx, 1, seq_ids, cu, mx, hv, sess.kv)
    sess.n_cache[0] = sess.n_seen[0] = T
    pos, sc = sess.read(0, 1)
    assert np.isnan(sc).sum() > 100
    kept = sess.select([0], [K])[0]
    assert list(kept) == O.select_kept(sc.astype(np.float64), K, 0, 128)
    sess.close()


def test_cluster_selection_on_a_30000_slot_cache(gpu_lib):
    """One 30,000-slot cache cut to 5,000 (slices of 3,750 slots, the
    metadata moved in one round), against the oracle on fp64 scores too."""
    model = W.small_model(93)
    T, K = 30000, 5000
    sess = Session(model, n_seq=2, kinds=KINDS, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=T, max_new=3000,
                   prefill=(0, 12), policies=(1, 2))
    for _ in range(T // 3000):
        sess.score_update([(0, 3000), (1, 3000)])
    pre = {b: sess.read(b, sess.policies[b]) for b in range(2)}
    kept = sess.select([0, 1], [K, K])
    sess.compact([0, 1])
    for b in range(2):
        pos, sc = pre[b]
        ref = OracleTrace(model, sess.dt.tabs, b, T, sess.policies[b])
        cond = ref.cond.get(sess.policies[b])
        check_selection(kept[b], pos, sc, ref.scores[sess.policies[b]][pos], K, sess.prefill[b], 128, 1,
                        None if cond is None else cond[pos])
        pos_after, _ = sess.read(b, sess.policies[b])
        np.testing.assert_array_equal(pos_after, pos[kept[b]])
        check_compaction(sess, b, pos_after)
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
