"""Device-side anomalies become sticky error codes, never faults.

Every case is an invalid input that the kernels' own bounds checks catch:
the offending work is skipped, epikv_get_error reports the code once, and the
context keeps working.  Nothing here traps, faults or waits on the GPU.
"""
import numpy as np
import pytest
import torch

from paper_2606_26472_gb300 import epikv as E
from synth import workloads as W

from .harness import Session

pytestmark = pytest.mark.gpu


def _session(kinds=E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV, layout=E.EPIKV_LAYOUT_PAGED, T=64, max_new=16):
    policies = (1, 2) if kinds == 3 else (kinds, kinds)
    return Session(W.small_model(31), n_seq=2, kinds=kinds, layout=layout, max_tokens=T, max_new=max_new,
                   prefill=(0, 0), policies=policies)


def _dev(x):
    return torch.tensor(x, dtype=torch.int32, device="cuda")


def test_oversized_batch_entry_is_rejected_on_the_device(gpu_lib):
    sess = _session()
    sess.score_update([(0, 8)])
    assert sess.error() == (E.EPIKV_OK, 0)
    seq_ids, _, _, hv = sess.append([(0, 8)])
    # the offsets claim 12 new tokens while the call declares at most 8
    E.epikv_score_update(sess.ctx, 1, seq_ids, _dev([0, 12]), 8, hv, sess.kv)
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_BATCH)
    assert sess.error() == (E.EPIKV_OK, 0)                        # cleared
    pos, _ = sess.read(0, 1)                                       # nothing was committed
    np.testing.assert_array_equal(pos, np.arange(8))
    sess.score_update([(0, 8)])                                    # the context still works
    assert sess.error() == (E.EPIKV_OK, 0)
    assert len(sess.read(0, 2)[0]) == 16
    sess.close()


def test_cache_capacity_overflow(gpu_lib):
    sess = _session(T=32, max_new=16)
    sess.score_update([(0, 16), (1, 16)])
    sess.score_update([(0, 16)])
    assert sess.error() == (E.EPIKV_OK, 0)
    seq_ids, cu, mx, hv = sess.append([(1, 8)])
    E.epikv_score_update(sess.ctx, 1, _dev([0]), cu, mx, hv, sess.kv)   # sequence 0 is full
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_CAPACITY)
    assert len(sess.read(0, 1)[0]) == 32
    sess.close()


def test_invalid_budget(gpu_lib):
    sess = _session()
    sess.score_update([(0, 16)])
    kept = torch.empty((1, 64), dtype=torch.int32, device="cuda")
    nk = torch.empty(1, dtype=torch.int32, device="cuda")
    E.epikv_select(sess.ctx, 1, _dev([0]), _dev([0]), None, kept, 64, nk)
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_BUDGET)
    assert int(nk.item()) == 16                                    # nothing evicted
    sess.close()


def test_block_id_outside_the_pool(gpu_lib):
    sess = _session(kinds=E.EPIKV_SCORE_LAGKV)
    sess.score_update([(0, 16)])
    seq_ids, cu, mx, hv = sess.append([(0, 8)])                   # rows written through the valid table
    bad = sess.cache.block_table.clone()
    bad[0, 1] = sess.cache.num_blocks + 5                          # slots 16..31 of sequence 0
    view = sess.cache.view(block_table=bad)
    E.epikv_score_update(sess.ctx, 1, seq_ids, cu, mx, hv, view)
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_SLOT)
    sess.close()


def test_kept_list_that_is_not_increasing(gpu_lib):
    sess = _session(kinds=E.EPIKV_SCORE_LAGKV)
    sess.score_update([(0, 16), (1, 16)])
    sess.score_update([(0, 16), (1, 16)])
    kept = torch.empty((2, 64), dtype=torch.int32, device="cuda")
    nk = torch.empty(2, dtype=torch.int32, device="cuda")
    ids = _dev([0, 1])
    E.epikv_select(sess.ctx, 2, ids, _dev([20, 20]), None, kept, 64, nk)
    torch.cuda.synchronize()
    assert sess.error() == (E.EPIKV_OK, 0)
    bad = kept.clone()
    bad[0, 19] = 3                                                 # a source before its destination
    E.epikv_compact(sess.ctx, 2, ids, bad, 64, sess.kv)
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_KEPT)
    sess.close()


def test_negative_layer_table_stride_is_rejected_on_the_host(gpu_lib):
    sess = _session(kinds=E.EPIKV_SCORE_LAGKV)
    seq_ids, cu, mx, hv = sess.append([(0, 8)])
    view = sess.cache.view()
    view.stride_table_layer = -1
    with pytest.raises(E.EpikvError) as err:
        E.epikv_score_update(sess.ctx, 1, seq_ids, cu, mx, hv, view)
    assert err.value.status == E.EPIKV_EINVAL
    assert sess.error() == (E.EPIKV_OK, 0)                        # nothing was enqueued
    sess.close()


def test_layer_budgets_that_break_the_nesting_are_reported(gpu_lib):
    """Per-layer budgets must stay fixed for a sequence: after layer 1 was cut
    to 20 tokens, giving it the largest budget asks it to keep tokens it no
    longer holds, which the selection reports instead of inventing rows."""
    model = W.small_model(32)
    sess = Session(model, n_seq=1, kinds=E.EPIKV_SCORE_BANDZ, layout=E.EPIKV_LAYOUT_CONTIGUOUS, max_tokens=96,
                   max_new=48, prefill=(0,), policies=(E.EPIKV_SCORE_BANDZ,), layer_budgets=1)
    sess.score_update([(0, 48)])
    sess.select([0], [[40, 20, 40, 40]])
    sess.compact([0])
    assert sess.error() == (E.EPIKV_OK, 0) and sess.n_layer[0] == [40, 20, 40, 40]
    sess.score_update([(0, 16)])
    sess.select([0], [[20, 40, 40, 40]])
    sess.compact([0])
    assert sess.error() == (E.EPIKV_EDEVICE, E.EPIKV_DEV_KEPT)
    assert sess.n_layer[0][1] <= 36                                # layer 1 kept only rows it holds
    sess.close()
