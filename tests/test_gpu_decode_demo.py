"""The decode-loop integration (examples/llama_decode.py) on a small
LLaMA-shaped random-weight model: the library's scores of the model's own
hidden states and K/V equal the fp64 oracle's, and the cache the model
attends over after each eviction holds exactly the kept tokens' rows."""
import os
import sys

import numpy as np
import pytest

from oracle import epikv_oracle as O
from paper_2606_26472_gb300 import epikv as E
from synth import gen

from .harness import assert_scores_close

pytestmark = pytest.mark.gpu

sys.path.insert(0, os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "examples"))


def test_random_llama_decode_with_eviction(gpu_lib):
    import llama_decode as D
    shape = D.small_shape()
    prompt, steps, K, slack = 8, 200, 96, 16
    r = D.decode(shape, batch=4, prompt=prompt, steps=steps, budget=K, slack=slack, record=True)
    assert E.epikv_get_error(r.ctx) == (E.EPIKV_OK, 0)
    T = prompt + steps
    assert r.evictions >= 4 * 5
    bt = r.cache.block_table.cpu().numpy()
    for b in range(4):
        ra = [gen.bf16_bits_to_f64(r.band_rows[(b, l)]) for l in shape.band_a]
        rb = [gen.bf16_bits_to_f64(r.band_rows[(b, l)]) for l in shape.band_b]
        Kr, Vr = r.kv_rows[b]
        ref = {E.EPIKV_SCORE_BANDZ: O.bandz_scores(ra, rb, 64),
               E.EPIKV_SCORE_LAGKV: O.lagkv_scores(gen.bf16_bits_to_f64(Kr), gen.bf16_bits_to_f64(Vr), 16)}
        for kind, sref in ref.items():
            pos, sc, n = E.epikv_read_slots(r.ctx, b, kind, 4096)
            pos = np.array(pos)
            assert n == r.n_cache[b] and len(pos) == n
            assert list(pos[:prompt]) == list(range(prompt))          # the prompt is never evicted
            assert np.all(np.diff(pos) > 0) and pos[-1] == T - 1
            assert_scores_close(sc, sref[pos], f"decode seq {b} kind {kind}")
        # the compacted cache holds the kept positions' rows, every layer and head
        k = r.cache.rows(0, b, np.arange(n), bt)
        v = r.cache.rows(1, b, np.arange(n), bt)
        from synth.device import as_u16
        np.testing.assert_array_equal(as_u16(k), Kr[pos])
        np.testing.assert_array_equal(as_u16(v), Vr[pos])
