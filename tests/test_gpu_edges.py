"""Edge cases of the path on the GPU: empty and ragged batches, budgets that
do not bind, prefill larger than the budget, prefill + recency >= K, NaN
scores, and calls with nothing to do."""
import numpy as np
import pytest
import torch

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from synth import gen, workloads as W

from .harness import OracleTrace, Session, assert_scores_close, check_compaction

pytestmark = pytest.mark.gpu

KINDS = E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV


def _dev(x):
    return torch.tensor(x, dtype=torch.int32, device="cuda")


def test_empty_batch_and_zero_token_entries(gpu_lib):
    sess = Session(W.small_model(41), n_seq=3, kinds=KINDS, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=96, max_new=8,
                   prefill=(0, 0, 0), policies=(1, 2, 1))
    E.epikv_score_update(sess.ctx, 0, None, None, 0, None, None)          # nothing to do
    E.epikv_step(sess.ctx, 0, None, None, 0, _dev([1]), None, None, sess.kv)
    refs = [OracleTrace(sess.m, sess.dt.tabs, b, 60, KINDS) for b in range(3)]
    # a ragged batch where some entries bring no token at all
    pattern = [(5, 0, 3), (0, 0, 8), (7, 8, 0), (2, 1, 1)]
    for step in range(12):
        counts = pattern[step % len(pattern)]
        entries = [(b, min(counts[b], 60 - sess.n_seen[b])) for b in range(3)]
        sess.score_update(entries)
    for b in range(3):
        for kind in (1, 2):
            pos, sc = sess.read(b, kind)
            assert_scores_close(sc, refs[b].scores[kind][pos], f"seq {b} kind {kind}")
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_budgets_that_do_not_bind_leave_everything(gpu_lib):
    sess = Session(W.small_model(42), n_seq=2, kinds=KINDS, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=80,
                   max_new=40, prefill=(0, 0), policies=(1, 2))
    sess.score_update([(0, 40), (1, 40)])
    before = [sess.read(b, 1)[0] for b in range(2)]
    kept = sess.select([0, 1], [40, 60])                 # n == K and n < K
    assert kept == {}
    kept = sess.select([0, 1], [20, 20], [40, 45])       # n does not exceed the trigger
    assert kept == {}
    sess.compact([0, 1])
    for b in range(2):
        np.testing.assert_array_equal(sess.read(b, 1)[0], before[b])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


@pytest.mark.parametrize("prefill,K", [(30, 20), (20, 24), (10, 12), (0, 1), (5, 6)])
def test_prefill_and_recency_against_the_budget(gpu_lib, prefill, K):
    """P > K keeps the whole prefill; P + R >= K shrinks the recency window;
    K = 1 keeps only the newest token (R = 0, M = 1 or the last slot)."""
    sess = Session(W.small_model(43), n_seq=1, kinds=KINDS, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=64,
                   max_new=64, prefill=(prefill,), policies=(1,))
    sess.score_update([(0, 50)])
    pos, sc = sess.read(0, 1)
    kept = sess.select([0], [K])[0]
    assert list(kept) == O.select_kept(sc.astype(np.float64), K, prefill, 128)
    assert len(kept) == max(K, min(prefill, 50))
    sess.compact([0])
    pos_after, _ = sess.read(0, 1)
    np.testing.assert_array_equal(pos_after, pos[kept])
    check_compaction(sess, 0, pos_after)
    sess.close()


def test_nan_scores_rank_lowest(gpu_lib):
    """A NaN in a band row makes g, and every z whose window holds it, NaN;
    the selection ranks NaN below every number, exactly as the oracle does."""
    model = W.small_model(44)
    T, K = 160, 70
    sess = Session(model, n_seq=1, kinds=E.EPIKV_SCORE_BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=T,
                   max_new=T, prefill=(0,), policies=(1,))
    seq_ids, cu, mx, hv = sess.append([(0, T)])
    sess.hid[0, 50, 3] = float("nan")                    # Band A layer, position 50
    E.epikv_score_update(sess.ctx, 1, seq_ids, cu, mx, hv, sess.kv)
    sess.n_cache[0] = sess.n_seen[0] = T
    pos, sc = sess.read(0, 1)
    # g(50), g(51) are NaN; windows of positions 50 .. 51 + 63 hold one of them
    assert np.isnan(sc[50]) and np.isnan(sc[114]) and not np.isnan(sc[49]) and not np.isnan(sc[115])
    kept = sess.select([0], [K])[0]
    assert list(kept) == O.select_kept(sc.astype(np.float64), K, 0, 128)
    assert not set(range(50, 115)) & set(kept[:-17])     # NaN candidates lose to every number
    sess.close()


@pytest.mark.parametrize("layer_budgets", [0, 1], ids=["token", "per_layer"])
def test_a_compaction_is_applied_once(gpu_lib, layer_budgets):
    """A selection's eviction is compacted once: a second epikv_compact (or
    one after a score update with no selection) leaves the cache alone."""
    model = W.small_model(45)
    sess = Session(model, n_seq=2, kinds=KINDS, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=120, max_new=100,
                   prefill=(0, 3), policies=(1, 2), layer_budgets=layer_budgets)
    budgets = [[40, 30, 50, 20], [60, 60, 25, 35]] if layer_budgets else [40, 60]

    def snapshot():
        return [np.stack(sess.cache_rows_u16(b, np.arange(sess.n_cache[b]))) for b in range(2)]

    sess.score_update([(0, 100), (1, 90)])
    sess.compact([0, 1])                     # nothing selected yet: nothing moves
    sess.select([0, 1], budgets)
    first = snapshot()
    sess.compact([0, 1])
    after = snapshot()
    sess.compact([0, 1])                     # the same eviction again: a no-op
    again = snapshot()
    for b in range(2):
        np.testing.assert_array_equal(after[b], again[b])
        assert not np.array_equal(first[b], after[b])    # the first compaction did move rows
        if layer_budgets:
            for l in range(model.num_layers):
                pos = sess.read_layer(b, l)
                k, v = sess.layer_rows_u16(b, l, np.arange(len(pos)))
                sp = gen.spike_flags(model, b, int(pos.max()) + 1)
                np.testing.assert_array_equal(k, gen.kv_rows(model, sess.dt.tabs, b, 0, pos, sp)[:, l])
        else:
            check_compaction(sess, b, sess.read(b, 1)[0])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
