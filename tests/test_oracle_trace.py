"""CPU checks of the harness's block-wise oracle traces: with row blocks far
smaller than a trace (and not a multiple of the lag), every score kind
equals the oracle's whole-trace functions on the whole trace's rows, so the
blocks and chunk look-backs add nothing of their own."""
import numpy as np

from oracle import epikv_oracle as O
from synth import gen, host, workloads as W

from . import harness as Hs


def _whole(model, tabs, seq, n, lag, w):
    pos = np.arange(n)
    sp = gen.spike_flags(model, seq, n)
    Kr = gen.bf16_bits_to_f64(gen.kv_rows(model, tabs, seq, 0, pos, sp))
    Vr = gen.bf16_bits_to_f64(gen.kv_rows(model, tabs, seq, 1, pos, sp))
    seg = gen.segment_index(model, seq, n)
    ra = [gen.bf16_bits_to_f64(gen.hidden_rows(model, tabs, seq, l, pos, seg)) for l in model.band_a]
    rb = [gen.bf16_bits_to_f64(gen.hidden_rows(model, tabs, seq, l, pos, seg)) for l in model.band_b]
    return {1: O.bandz_scores(ra, rb, w), 2: O.lagkv_scores(Kr, Vr, lag, w=w), 4: O.hsvar_scores(ra, rb, w),
            8: O.kv_variance_scores(Kr, w), 16: O.kv_variance_scores(Vr, w), 32: O.lag_key_scores(Kr, lag, w=w)}


def test_blockwise_traces_equal_whole_trace_oracle(monkeypatch):
    monkeypatch.setattr(Hs, "ROW_BLOCK", 37)
    cases = ((W.small_model(5), 0, 230, 16, 64), (W.small_model(6), 2, 181, 5, 20),
             (gen.TraceModel(0xE91C00B7), 1, 90, 16, 64))
    for model, seq, n, lag, w in cases:
        tabs = gen.make_tables(model)
        tr = Hs.OracleTrace(model, tabs, seq, n, 63, z_window=w, lag=lag, lag_window=w)
        ref = _whole(model, tabs, seq, n, lag, w)
        for kind, s in ref.items():
            np.testing.assert_array_equal(tr.scores[kind], s, err_msg=f"kind {kind}")
        # the band-z condition numbers come from the same g traces
        seg = gen.segment_index(model, seq, n)
        pos = np.arange(n)
        ra = [gen.bf16_bits_to_f64(host.hidden_rows(model, tabs, seq, l, pos, seg)) for l in model.band_a]
        rb = [gen.bf16_bits_to_f64(host.hidden_rows(model, tabs, seq, l, pos, seg)) for l in model.band_b]
        np.testing.assert_array_equal(tr.cond[1], Hs.bandz_condition(ra, rb, w))
        assert tr.cond.get(2) is None
