"""Chunk-level selection on the GPU (the chunk-level scoring the paper names
as future work, Sec. 5): the one-call step path equals the split calls bit
for bit, each event's kept list equals the oracle's on the GPU's own scores,
and the degenerate cases (one chunk holding every candidate, a NaN inside a
chunk) behave as the oracle's rule says."""
import numpy as np
import pytest

from paper_2606_26472_gb300 import epikv as E
from synth import workloads as W

from .harness import Session, check_compaction, oracle_kept

pytestmark = pytest.mark.gpu

BANDZ, LAGKV = E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV


def test_step_equals_split_calls_and_the_oracle(gpu_lib):
    model = W.small_model(61)
    C = 8
    kw = dict(n_seq=3, kinds=BANDZ | LAGKV, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=200, max_new=24,
              prefill=(4, 0, 0), policies=(BANDZ, LAGKV, BANDZ), select_chunk=C)
    a, b = Session(model, **kw), Session(model, **kw)
    budgets, slack = [90, 64, 120], 10
    triggers = [k + slack for k in budgets]
    pattern = (24, 3, 17, 9)
    events = 0
    for step in range(30):
        entries = [(s, pattern[(s + step) % len(pattern)]) for s in range(3)]
        a.step(entries, budgets, triggers)
        b.score_update(entries)
        pre = {s: b.read(s, b.policies[s]) for s in range(3)}
        kept = b.select(list(range(3)), budgets, triggers)
        b.compact(list(range(3)))
        for s, kl in kept.items():
            events += 1
            pos, sc = pre[s]
            assert list(kl) == oracle_kept(sc, pos, budgets[s], b.prefill[s], 128, C)
        for s in range(3):
            assert a.n_cache[s] == b.n_cache[s]
            for kind in (BANDZ, LAGKV):
                pa, sa = a.read(s, kind)
                pb, sb = b.read(s, kind)
                np.testing.assert_array_equal(pa, pb)
                np.testing.assert_array_equal(sa.view(np.uint32), sb.view(np.uint32))
    assert events >= 9
    for s in range(3):
        n = a.n_cache[s]
        ka, va = a.cache_rows_u16(s, np.arange(n))
        kb, vb = b.cache_rows_u16(s, np.arange(n))
        np.testing.assert_array_equal(ka, kb)
        np.testing.assert_array_equal(va, vb)
        check_compaction(a, s, a.read(s, BANDZ)[0])
    assert a.error() == b.error() == (E.EPIKV_OK, 0)
    a.close()
    b.close()


def test_one_chunk_holding_every_candidate_keeps_its_lowest_slots(gpu_lib):
    T, K, P = 300, 100, 5                      # R = 25, M = 70
    sess = Session(W.small_model(62), n_seq=1, kinds=BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=T,
                   max_new=T, prefill=(P,), policies=(BANDZ,), select_chunk=65536)
    sess.score_update([(0, T)])
    pos, sc = sess.read(0, BANDZ)
    kept = sess.select([0], [K])[0]
    assert list(kept) == list(range(P + 70)) + list(range(T - 25, T))
    assert list(kept) == oracle_kept(sc, pos, K, P, 128, 65536)
    sess.compact([0])
    check_compaction(sess, 0, sess.read(0, BANDZ)[0])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_a_nan_makes_its_whole_chunk_rank_lowest(gpu_lib):
    """A NaN band row makes the scores of positions 50 .. 114 NaN (their z
    windows hold a NaN g); with 8-position chunks, chunks 6 .. 14 (positions
    48 .. 119) have NaN means and lose to every other chunk, including the
    finite scores at positions 48, 49 and 115 .. 119."""
    T, K, C = 160, 70, 8                       # R = 17, M = 53 < 71 finite-chunk slots
    sess = Session(W.small_model(44), n_seq=1, kinds=BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=T,
                   max_new=T, prefill=(0,), policies=(BANDZ,), select_chunk=C)
    seq_ids, cu, mx, hv = sess.append([(0, T)])
    sess.hid[0, 50, 3] = float("nan")
    E.epikv_score_update(sess.ctx, 1, seq_ids, cu, mx, hv, sess.kv)
    sess.n_cache[0] = sess.n_seen[0] = T
    pos, sc = sess.read(0, BANDZ)
    assert np.isnan(sc[50]) and np.isnan(sc[114]) and not np.isnan(sc[49]) and not np.isnan(sc[115])
    kept = sess.select([0], [K])[0]
    assert list(kept) == oracle_kept(sc, pos, K, 0, 128, C)
    assert not set(range(48, 120)) & set(kept[:-17])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
