"""epikv_set_kernel_events: every kernel a context's calls launch is bracketed
by two of the caller's events, in launch order, with the runtime's name of
the kernel; the step's results are unchanged by the timing, and a capacity
smaller than the launches records the first ones only."""
import numpy as np
import pytest
import torch

from paper_2606_26472_gb300 import epikv as E
from synth import workloads as W

from .harness import Session

pytestmark = pytest.mark.gpu


def _run(timed):
    model = W.small_model(77)
    kinds = E.EPIKV_SCORE_LAGKV
    sess = Session(model, n_seq=2, kinds=kinds, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=96, max_new=32,
                   prefill=(0, 0), policies=(kinds, kinds))
    recs = []
    for step in range(4):
        if timed and step == 3:
            kc = E.KernelClock(sess.ctx, 16)
            kc.start()
            sess.step([(0, 32), (1, 32)], [64, 64], [64, 64])
            recs = kc.stop()
        else:
            sess.step([(0, 32), (1, 32)], [64, 64], [64, 64])
    out = [sess.read(b, kinds) for b in range(2)]
    k, v = sess.cache_rows_u16(0, np.arange(64))
    assert sess.error() == (E.EPIKV_OK, 0)
    sess.close()
    return recs, out, k, v


def test_kernel_events_bracket_every_launch_in_order(gpu_lib):
    recs, out, k, v = _run(True)
    names = [E.kernel_short_name(n) for n, _ in recs]
    # the step after the caches are full: score (partial + finalize), select, stash, copy, marker
    assert names == ["lagkv_partial_kernel", "score_finalize_kernel", "select_kernel", "compact_stash_kernel",
                     "compact_kernel", "compact_consumed_kernel"], names
    assert all(ms > 0 for _, ms in recs)
    recs0, out0, k0, v0 = _run(False)
    for (p, s), (p0, s0) in zip(out, out0):   # timing changes nothing
        np.testing.assert_array_equal(p, p0)
        np.testing.assert_array_equal(s, s0)
    np.testing.assert_array_equal(k, k0)
    np.testing.assert_array_equal(v, v0)


def test_kernel_events_capacity_records_the_first_launches(gpu_lib):
    model = W.small_model(78)
    kinds = E.EPIKV_SCORE_BANDZ
    sess = Session(model, n_seq=1, kinds=kinds, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=64, max_new=16,
                   prefill=(0,), policies=(kinds,))
    kc = E.KernelClock(sess.ctx, 2)
    kc.start()
    sess.score_update([(0, 16)])
    sess.score_update([(0, 16)])
    recs = kc.stop()
    assert [E.kernel_short_name(n) for n, _ in recs] == ["bandz_g_kernel", "score_finalize_kernel"]
    sess.close()
