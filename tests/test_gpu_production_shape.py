"""Element-wise parity at the production model shape: 32 layers x 8 KV heads x
128 dims (16 lanes per head: the lagkv_partial_kernel<16> and
token_kernel<16> instances the 32k workload runs) and hidden 4096 with the
15 band layers 7..13 / 18..25.  Two sequences of 1,536 tokens, every score
kind, both K/V layouts, evictions to K = 512:

* chunked calls: sequence 0 takes 128 tokens per call (whole Lag-KV chunks
  and 8-token segments); sequence 1 takes a ragged pattern (1, 7, 128, 100,
  16, 3, 64, 33 tokens) whose calls start and end inside lag chunks and
  segments, with 16 prefill tokens;
* one-token calls (the decode-step kernels, both halves of a 256-thread CTA
  carrying one layer's K and V streams).

Every position's score of every kind is compared with the fp64 oracle right
after the call that scores it; every eviction's kept list is checked exactly
against the oracle's selection on the GPU's own scores and, against the fp64
scores, up to threshold ties; compacted rows are compared byte for byte with
the generator's rows of the kept positions."""
import numpy as np
import pytest

from paper_2606_26472_gb300 import epikv as E
from synth import gen

from .harness import ALL_KINDS, OracleTrace, Session, check_compaction, check_compaction_sampled, check_selection

pytestmark = pytest.mark.gpu

MODEL = gen.TraceModel(0xE91C00B7)       # the full 32 x 8 x 128, hidden 4096, bands 7..13 / 18..25 shape
T = 1536
KINDS = 63
K = 512
PREFILL = (0, 16)
RAGGED = (1, 7, 128, 100, 16, 3, 64, 33)


@pytest.fixture(scope="module")
def refs():
    tabs = gen.make_tables(MODEL)
    return [OracleTrace(MODEL, tabs, b, T, KINDS) for b in range(2)]


def _drive(refs, layout, policies, chunk_of, slack, max_new, kinds=KINDS):
    """Decode both sequences to T tokens; chunk_of(b, call) = tokens of
    sequence b in that call."""
    sess = Session(MODEL, n_seq=2, kinds=kinds, layout=layout, max_tokens=K + slack + max_new + 1, max_new=max_new,
                   prefill=PREFILL, policies=policies)
    rng = np.random.default_rng(7)
    checked = [0, 0]          # positions whose scores were compared, per sequence
    events = 0
    call = 0
    while any(sess.n_seen[b] < T for b in range(2)):
        entries = [(b, min(chunk_of(b, call), T - sess.n_seen[b])) for b in range(2) if sess.n_seen[b] < T]
        call += 1
        before = {b: sess.n_cache[b] for b, _ in entries}
        sess.score_update(entries)
        pre = {}
        for b, n in entries:
            for kind in (k for k in ALL_KINDS if kinds & k):
                pos, sc = sess.read(b, kind)
                new = slice(before[b], before[b] + n)
                np.testing.assert_array_equal(pos[new], np.arange(sess.n_seen[b] - n, sess.n_seen[b]))
                refs[b].check(kind, pos[new], sc[new], f"{layout=} seq {b} kind {kind} call {call}")
                if kind == policies[b]:
                    pre[b] = (pos, sc)
            checked[b] += n
        seqs = [b for b, _ in entries]
        if not any(sess.n_cache[b] > K + slack for b in seqs):
            continue
        kept = sess.select(seqs, [K] * len(seqs), [K + slack] * len(seqs))
        sess.compact(seqs)
        for b, kl in kept.items():
            pos, sc = pre[b]
            cond = refs[b].cond.get(policies[b])
            check_selection(kl, pos, sc, refs[b].scores[policies[b]][pos], K, PREFILL[b], 128, 1,
                            None if cond is None else cond[pos])
            pos_after, _ = sess.read(b, policies[b])
            np.testing.assert_array_equal(pos_after, pos[kl])
            if events < 2:
                check_compaction(sess, b, pos_after)
            else:
                check_compaction_sampled(sess, b, pos_after, 48, rng)
            events += 1
    assert checked == [T, T]
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
    return events


@pytest.mark.parametrize("layout", [E.EPIKV_LAYOUT_PAGED, E.EPIKV_LAYOUT_CONTIGUOUS], ids=["paged", "contiguous"])
def test_production_shape_chunked_calls(gpu_lib, refs, layout):
    policies = (E.EPIKV_SCORE_LAGKV, E.EPIKV_SCORE_LAGKEY) if layout else (E.EPIKV_SCORE_KVKEY, E.EPIKV_SCORE_BANDZ)
    events = _drive(refs, layout, policies, lambda b, c: 128 if b == 0 else RAGGED[c % len(RAGGED)], 127, 128)
    assert events >= 12


@pytest.mark.parametrize("layout", [E.EPIKV_LAYOUT_PAGED, E.EPIKV_LAYOUT_CONTIGUOUS], ids=["paged", "contiguous"])
def test_production_shape_one_token_calls(gpu_lib, refs, layout):
    policies = (E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV) if layout else (E.EPIKV_SCORE_KVVAL, E.EPIKV_SCORE_HSVAR)
    events = _drive(refs, layout, policies, lambda b, c: 1, 64, 1)
    assert events >= 25


def test_production_shape_one_token_calls_band_kinds_only(gpu_lib, refs):
    """One-token calls with only the band kinds take the fused band-z decode
    kernel (bandz_token_kernel, 2 row vectors per thread at hidden 4096)."""
    kinds = E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_HSVAR
    events = _drive(refs, E.EPIKV_LAYOUT_PAGED, (E.EPIKV_SCORE_HSVAR, E.EPIKV_SCORE_BANDZ), lambda b, c: 1, 64, 1,
                    kinds)
    assert events >= 25
