"""The compaction's two work splits on the GPU.

The moved rows of all streams are cut into one equal chunk per CTA, the
sources a chunk still reads from later chunks' regions copied aside first,
when those rows fit the 128-row stash: when every evicting entry's largest
shift (its last kept slot minus its new length minus one) is at most 128, or
when no chunk is longer than 128 rows (ceil(total moved rows / 304 CTAs));
otherwise each (entry, layer, K|V) stream is one unit.  Both must leave every
kept row in its slot, byte for byte: these cases reach the split through
either bound or neither, give far fewer rows than CTAs, hold fewer slots than
the stash, and mix entries of both kinds in one batch."""
import numpy as np
import pytest
import torch

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from synth import gen, workloads as W

from .harness import Session, check_compaction, check_compaction_sampled

pytestmark = pytest.mark.gpu


def _rows(sess, b, n):
    """Every layer's K and V rows of slots 0..n-1 (device gathers)."""
    slots = np.arange(n)
    return sess.cache.rows(0, b, slots, sess.bt_host).clone(), sess.cache.rows(1, b, slots, sess.bt_host).clone()


def _evict_and_check(sess, budgets, generator_check=True, sampled=0):
    """Select and compact every entry; each entry's compacted slot i holds,
    byte for byte, what slot kept[i] held before (compared on the device over
    the whole cache), and those are the generator's rows of the kept
    positions (all of them, or `sampled` random slots)."""
    seqs = list(range(len(budgets)))
    pre = {b: sess.read(b, sess.policies[b]) for b in seqs}
    before = {b: _rows(sess, b, sess.n_cache[b]) for b in seqs}
    kept = sess.select(seqs, budgets)
    sess.compact(seqs)
    rng = np.random.default_rng(len(seqs))
    for b in seqs:
        pos, sc = pre[b]
        if len(pos) <= budgets[b]:
            assert b not in kept
            after = _rows(sess, b, len(pos))
            assert all(torch.equal(x.view(torch.int16), y.view(torch.int16)) for x, y in zip(after, before[b]))
            continue
        exp = O.select_kept(sc.astype(np.float64), budgets[b], sess.prefill[b], sess.recency_cap)
        assert list(kept[b]) == exp
        pos_after, _ = sess.read(b, sess.policies[b])
        np.testing.assert_array_equal(pos_after, pos[kept[b]])
        after = _rows(sess, b, len(kept[b]))
        idx = torch.as_tensor(kept[b], device=after[0].device)
        for x, y in zip(after, before[b]):
            assert torch.equal(x.view(torch.int16), y.index_select(0, idx).view(torch.int16)), f"seq {b}"
        if generator_check:
            check_compaction(sess, b, pos_after)
        elif sampled:
            check_compaction_sampled(sess, b, pos_after, sampled, rng)
    assert sess.error() == (E.EPIKV_OK, 0)
    return kept


@pytest.mark.parametrize("layout", [E.EPIKV_LAYOUT_PAGED, E.EPIKV_LAYOUT_CONTIGUOUS])
@pytest.mark.parametrize("evict", [1, 128, 129, 300])
def test_one_full_size_sequence_either_side_of_the_stash_bound(gpu_lib, layout, evict):
    """One 32-layer sequence of 600 tokens cut by `evict` slots: its largest
    shift is `evict`, within the stash up to 128; above it the chunks (at
    most 64 x 600 / 304 < 128 rows) are the bound that admits the split."""
    model = gen.TraceModel(0xC0A1 + evict)
    sess = Session(model, n_seq=1, kinds=E.EPIKV_SCORE_LAGKV, layout=layout, max_tokens=640, max_new=200,
                   prefill=(0,), policies=(E.EPIKV_SCORE_LAGKV,))
    for _ in range(3):
        sess.score_update([(0, 200)])
    kept = _evict_and_check(sess, [600 - evict], generator_check=False, sampled=48)
    shift = int(kept[0][-1]) - (len(kept[0]) - 1)
    assert shift == evict
    sess.close()


def test_fewer_moved_rows_than_ctas(gpu_lib):
    """A long protected prefill leaves a handful of candidates: a few rows
    move per stream, most chunks are empty and the others are one row long,
    ending inside a stream."""
    sess = Session(W.small_model(0xC0A2), n_seq=2, kinds=E.EPIKV_SCORE_BANDZ, layout=E.EPIKV_LAYOUT_PAGED,
                   max_tokens=64, max_new=64, prefill=(40, 44), policies=(1, 1))
    sess.score_update([(0, 50), (1, 50)])
    kept = _evict_and_check(sess, [48, 49])
    assert all(int(kept[b][-1]) - (len(kept[b]) - 1) <= 2 for b in kept)
    sess.close()


@pytest.mark.parametrize("layout", [E.EPIKV_LAYOUT_PAGED, E.EPIKV_LAYOUT_CONTIGUOUS])
def test_cache_smaller_than_the_stash(gpu_lib, layout):
    """40 slots (the stash holds min(128, T) = 40 rows per CTA) cut to 10:
    shifts up to 30, balanced split."""
    sess = Session(W.small_model(0xC0A3), n_seq=3, kinds=E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV, layout=layout,
                   max_tokens=40, max_new=40, prefill=(0, 3, 0), policies=(1, 2, 1))
    sess.score_update([(0, 40), (1, 37), (2, 25)])
    _evict_and_check(sess, [10, 12, 20])
    sess.close()


@pytest.mark.parametrize("big", [False, True])
def test_batch_of_mixed_entries(gpu_lib, big):
    """Seven entries with different first moved slots and lengths, one of
    them untouched; with `big`, one entry's shift (200) exceeds the stash and
    the short chunks (fewer than 8 x 1,800 / 304 rows) admit the split."""
    n = 7
    sess = Session(W.small_model(0xC0A4 + big), n_seq=n, kinds=E.EPIKV_SCORE_LAGKV, layout=E.EPIKV_LAYOUT_PAGED,
                   max_tokens=512, max_new=256, prefill=(0, 17, 0, 64, 0, 5, 0),
                   policies=(E.EPIKV_SCORE_LAGKV,) * n)
    lens = [500, 300, 480, 260, 129, 400, 90]
    sess.score_update([(b, min(256, lens[b])) for b in range(n)])
    sess.score_update([(b, lens[b] - 256) for b in range(n) if lens[b] > 256])
    budgets = [300 if big else 420, 290, 470, 200, 100, 384, 120]
    kept = _evict_and_check(sess, budgets)
    shifts = [int(kept[b][-1]) - (len(kept[b]) - 1) for b in sorted(kept)]
    assert (max(shifts) > 128) == big
    assert 6 not in kept     # 90 tokens under a budget of 120
    sess.close()


def test_split_over_repeated_decode_evictions(gpu_lib):
    """Per-token decode with eviction whenever a cache exceeds K + 8: the
    entries evict at different steps, one or two at a time, each with a
    shift of nine slots, over many rounds."""
    n = 4
    sess = Session(W.small_model(0xC0A5), n_seq=n, kinds=E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV,
                   layout=E.EPIKV_LAYOUT_PAGED, max_tokens=96, max_new=64, prefill=(0, 4, 0, 0),
                   policies=(1, 2, 2, 1))
    K = [48, 56, 64, 40]
    sess.score_update([(0, 44), (1, 50), (2, 60), (3, 33)])
    events = 0
    for _ in range(40):
        sess.score_update([(b, 1) for b in range(n)])
        over = [b for b in range(n) if sess.n_cache[b] > K[b] + 8]
        if over:
            for b in over:
                pos, sc = sess.read(b, sess.policies[b])
                kept = sess.select([b], [K[b]])[b]
                assert list(kept) == O.select_kept(sc.astype(np.float64), K[b], sess.prefill[b], 128)
                sess.compact([b])
                pos_after, _ = sess.read(b, sess.policies[b])
                np.testing.assert_array_equal(pos_after, pos[kept])
                check_compaction(sess, b, pos_after)
                events += 1
    assert events >= 8
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


@pytest.mark.parametrize("evict", [100, 300])
def test_full_size_batch_past_both_bounds(gpu_lib, evict):
    """Three 32-layer sequences of 1,200 tokens cut by `evict` slots: about
    3 x 64 x 900 moved rows make chunks of ~570 rows, so a shift of 300
    leaves the balanced split for the per-stream units, and 100 keeps it."""
    n = 3
    model = gen.TraceModel(0xC0A6 + evict)
    sess = Session(model, n_seq=n, kinds=E.EPIKV_SCORE_LAGKV, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=1216,
                   max_new=400, prefill=(0,) * n, policies=(E.EPIKV_SCORE_LAGKV,) * n)
    for _ in range(3):
        sess.score_update([(b, 400) for b in range(n)])
    kept = _evict_and_check(sess, [1200 - evict] * n, generator_check=False, sampled=24)
    shifts = [int(kept[b][-1]) - (len(kept[b]) - 1) for b in range(n)]
    moved = sum(len(kept[b]) - next(i for i, k in enumerate(kept[b]) if k != i) for b in range(n))
    assert max(shifts) == evict
    assert -(-moved * 64 // 304) > 128
    sess.close()
