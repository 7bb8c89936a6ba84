"""The K/V kernels at the edges of the head shapes the library accepts: one
lane per head (d = 8, 32 heads), a full warp per head and the widest row
(d = 256, 8 heads: 256 lanes, 4 KiB rows), and a single head.  Every score
kind on a decode with evictions: scores against the fp64 oracle, kept lists
against the oracle's selection on the GPU's own scores, compacted rows
against the generator."""
import numpy as np
import pytest

from paper_2606_26472_gb300 import epikv as E
from synth import gen

from .harness import ALL_KINDS, OracleTrace, Session, assert_scores_close, check_compaction, check_selection

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("H,d,layout", [(32, 8, E.EPIKV_LAYOUT_PAGED), (8, 256, E.EPIKV_LAYOUT_CONTIGUOUS),
                                        (1, 64, E.EPIKV_LAYOUT_PAGED)], ids=["h32_d8", "h8_d256", "h1_d64"])
def test_head_shape_edges(gpu_lib, H, d, layout):
    model = gen.TraceModel(0xE91C0100 + H * d, num_layers=3, hidden=256, num_kv_heads=H, head_dim=d,
                           band_a=(1,), band_b=(2,))
    kinds = 63
    policies = (E.EPIKV_SCORE_LAGKV, E.EPIKV_SCORE_KVVAL)
    lengths, budgets, chunks, slack = (150, 130), (60, 48), (9, 20), 8
    sess = Session(model, n_seq=2, kinds=kinds, layout=layout, max_tokens=max(budgets) + slack + max(chunks) + 1,
                   max_new=max(chunks), prefill=(0, 3), policies=policies)
    refs = [OracleTrace(model, sess.dt.tabs, b, lengths[b], kinds) for b in range(2)]
    events, step = 0, 0
    while any(sess.n_seen[b] < lengths[b] for b in range(2)):
        entries = [(b, min(chunks[(b + step) % 2], lengths[b] - sess.n_seen[b])) for b in range(2)
                   if sess.n_seen[b] < lengths[b]]
        step += 1
        before = {b: sess.n_cache[b] for b, _ in entries}
        sess.score_update(entries)
        pre = {}
        for b, n in entries:
            for kind in ALL_KINDS:
                pos, sc = sess.read(b, kind)
                new = slice(before[b], before[b] + n)
                assert_scores_close(sc[new], refs[b].scores[kind][pos[new]], f"H{H} d{d} seq {b} kind {kind}")
                if kind == policies[b]:
                    pre[b] = (pos, sc)
        seqs = [b for b, _ in entries]
        kept = sess.select(seqs, [budgets[b] for b in seqs], [budgets[b] + slack for b in seqs])
        sess.compact(seqs)
        for b, kl in kept.items():
            events += 1
            pos, sc = pre[b]
            check_selection(kl, pos, sc, refs[b].scores[policies[b]][pos], budgets[b], sess.prefill[b], 128)
            pos_after, _ = sess.read(b, policies[b])
            np.testing.assert_array_equal(pos_after, pos[kl])
            check_compaction(sess, b, pos_after)
    assert events >= 6
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
