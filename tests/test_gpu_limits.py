"""The path at the limits of its configuration: an 8192-wide hidden state (four
16-byte vectors per thread in the g kernels, multi-token and one-token
calls), 32 band layers with a 1,024-token z window and a 1,024-token K/V
window (the finalize kernel's largest shared-memory staging), and a batch of
300 sequences in one call.  Scores against the fp64 oracle, kept lists
against the oracle's selection on the GPU's own scores, compacted rows
against the generator."""
import numpy as np
import pytest

from paper_2606_26472_gb300 import epikv as E
from synth import gen

from .harness import OracleTrace, Session, check_compaction, check_selection

pytestmark = pytest.mark.gpu

BANDZ, LAGKV, HSVAR = E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV, E.EPIKV_SCORE_HSVAR


@pytest.mark.parametrize("chunk", [1, 37], ids=["one_token_calls", "multi_token_calls"])
def test_widest_hidden_state(gpu_lib, chunk):
    model = gen.TraceModel(0xE91C0201, num_layers=3, hidden=8192, num_kv_heads=1, head_dim=8,
                           band_a=(0,), band_b=(1, 2))
    T = 150
    kinds = BANDZ | HSVAR
    sess = Session(model, n_seq=2, kinds=kinds, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=T, max_new=chunk,
                   prefill=(0, 0), policies=(BANDZ, HSVAR))
    refs = [OracleTrace(model, sess.dt.tabs, b, T, kinds) for b in range(2)]
    while sess.n_seen[0] < T:
        n = min(chunk, T - sess.n_seen[0])
        sess.score_update([(0, n), (1, n)])
    for b in range(2):
        for kind in (BANDZ, HSVAR):
            pos, sc = sess.read(b, kind)
            refs[b].check(kind, pos, sc, f"D=8192 seq {b} kind {kind}")
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_largest_windows_and_band_count(gpu_lib):
    model = gen.TraceModel(0xE91C0202, num_layers=32, hidden=64, num_kv_heads=1, head_dim=8,
                           band_a=tuple(range(16)), band_b=tuple(range(16, 32)))
    T, K = 1300, 700
    kinds = BANDZ | HSVAR | LAGKV
    sess = Session(model, n_seq=1, kinds=kinds, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=T, max_new=400,
                   prefill=(3,), policies=(BANDZ,), z_window=1024, lag_window=1024)
    ref = OracleTrace(model, sess.dt.tabs, 0, T, kinds, z_window=1024, lag_window=1024)
    while sess.n_seen[0] < T:
        sess.score_update([(0, min(400, T - sess.n_seen[0]))])
    pos, sc = sess.read(0, BANDZ)
    for kind in (BANDZ, HSVAR, LAGKV):
        p_, s_ = sess.read(0, kind)
        ref.check(kind, p_, s_, f"32 bands, windows 1024, kind {kind}")
    kept = sess.select([0], [K])[0]
    sess.compact([0])
    check_selection(kept, pos, sc, ref.scores[BANDZ][pos], K, 3, 128, 1, ref.cond[BANDZ][pos])
    check_compaction(sess, 0, sess.read(0, BANDZ)[0])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


@pytest.mark.parametrize("kinds", [BANDZ | HSVAR, BANDZ | HSVAR | LAGKV], ids=["band-kinds", "with-lagkv"])
def test_largest_windows_and_band_count_one_token_calls(gpu_lib, kinds):
    """The decode-step kernels at the limits: 32 band layers (the last CTA
    combines 32 per-band z values and window means over all 32 lanes) and
    windows of 1,024, one token per call past position 1,100, every score
    compared with the fp64 oracle (bandz_token_kernel for the band kinds
    alone, token_kernel with Lag-KV)."""
    model = gen.TraceModel(0xE91C0204, num_layers=32, hidden=64, num_kv_heads=1, head_dim=8,
                           band_a=tuple(range(16)), band_b=tuple(range(16, 32)))
    T = 1180
    sess = Session(model, n_seq=1, kinds=kinds, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=T, max_new=400,
                   prefill=(3,), policies=(BANDZ,), z_window=1024, lag_window=1024)
    ref = OracleTrace(model, sess.dt.tabs, 0, T, kinds, z_window=1024, lag_window=1024)
    while sess.n_seen[0] < 1100:
        sess.score_update([(0, min(400, 1100 - sess.n_seen[0]))])
    while sess.n_seen[0] < T:
        sess.score_update([(0, 1)])
    for kind in (k for k in (BANDZ, HSVAR, LAGKV) if kinds & k):
        p_, s_ = sess.read(0, kind)
        ref.check(kind, p_, s_, f"32 bands, windows 1024, one-token calls, kind {kind}")
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


def test_three_hundred_sequences_in_one_call(gpu_lib):
    model = gen.TraceModel(0xE91C0203, num_layers=2, hidden=64, num_kv_heads=1, head_dim=16,
                           band_a=(0,), band_b=(1,))
    S, T, K = 300, 48, 20
    kinds = BANDZ | LAGKV
    policies = [BANDZ if b % 2 else LAGKV for b in range(S)]
    sess = Session(model, n_seq=S, kinds=kinds, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=T, max_new=T,
                   prefill=[b % 3 for b in range(S)], policies=policies, block_size=4)
    sess.score_update([(b, T - (b % 7)) for b in range(S)])
    pre = {b: sess.read(b, policies[b]) for b in range(S)}
    kept = sess.select(list(range(S)), [K + (b % 5) for b in range(S)])
    sess.compact(list(range(S)))
    assert len(kept) == S
    rng = np.random.default_rng(3)
    for b in sorted(rng.choice(S, size=40, replace=False)):
        pos, sc = pre[b]
        ref = OracleTrace(model, sess.dt.tabs, b, T - (b % 7), kinds)
        ref.check(policies[b], pos, sc, f"seq {b}")
        check_selection(kept[b], pos, sc, ref.scores[policies[b]][pos], K + (b % 5), b % 3, 128, 1,
                        ref.cond[BANDZ][pos] if policies[b] == BANDZ else None)
        check_compaction(sess, b, sess.read(b, policies[b])[0])
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()


@pytest.mark.parametrize("hidden,bands", [(8192, 32), (4096, 32), (4096, 15), (2048, 17)],
                         ids=["D8192_32bands", "D4096_32bands", "D4096_15bands", "D2048_17bands"])
def test_band_decode_kernel_widths_and_band_counts(gpu_lib, hidden, bands):
    """The band-only decode kernel at the hidden widths that change its
    per-thread vectors (one, two or four 16-byte vectors of each row) with up
    to 32 band layers (the last CTA of a sequence combines 32 z values).
    One-token calls are compared with the fp64 oracle and, bit for bit, with
    the same trace scored in 40-token calls."""
    nA = bands // 2
    model = gen.TraceModel(0xE91C0205 + hidden + bands, num_layers=bands, hidden=hidden, num_kv_heads=1,
                           head_dim=8, band_a=tuple(range(nA)), band_b=tuple(range(nA, bands)))
    T = 120
    kinds = BANDZ | HSVAR
    out = []
    for chunk in (1, 40):
        sess = Session(model, n_seq=2, kinds=kinds, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=T, max_new=chunk,
                       prefill=(0, 0), policies=(BANDZ, HSVAR))
        while sess.n_seen[0] < T:
            n = min(chunk, T - sess.n_seen[0])
            sess.score_update([(0, n), (1, n)])
        out.append([[sess.read(b, k)[1] for k in (BANDZ, HSVAR)] for b in range(2)])
        if chunk == 1:
            for b in range(2):
                ref = OracleTrace(model, sess.dt.tabs, b, T, kinds)
                for k in (BANDZ, HSVAR):
                    pos, sc = sess.read(b, k)
                    ref.check(k, pos, sc, f"D={hidden}, {bands} bands, seq {b}, kind {k}")
        assert sess.error() == (E.EPIKV_OK, 0)
        sess.close()
    for b in range(2):
        for one, many in zip(out[0][b], out[1][b]):
            np.testing.assert_array_equal(one, many)
