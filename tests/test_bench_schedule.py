"""Host logic of bench.py's decode-window workloads (no GPU): the ragged
64-sequence schedule evicts every sequence exactly once per 65 calls, one
sequence per call but one, and never writes past a cache's capacity; the
8 x 8k schedule evicts every sequence at every call."""
import numpy as np
import pytest

import bench
from synth import workloads as W


def _setup(i):
    wl = W.config(i)
    budgets = np.array(wl.budgets, dtype=np.int64)
    slack = wl.trigger_slack[0]
    cycle = slack + 1
    n0 = budgets + ((np.arange(wl.n_seq) * 29) % cycle if wl.chunk == 1 else 0)
    return wl, budgets, slack, cycle, n0


def test_ragged_schedule_spreads_the_evictions():
    wl, budgets, slack, cycle, n0 = _setup(5)
    pos, slots, ev, n_end = bench.window_schedule(n0, budgets, slack, wl.chunk, 4 * cycle)
    assert len(set((n0 - budgets).tolist())) == wl.n_seq     # 64 distinct phases in a 65-call cycle
    per_cycle = ev.reshape(4, cycle).sum(axis=1)
    assert (per_cycle == wl.n_seq).all()                  # every sequence once per cycle
    assert ev.max() == 1                                  # at most one sequence per call
    cap = budgets + cycle                                  # slots 0 .. K + slack
    assert (slots.reshape(4 * cycle, wl.n_seq) < cap[None, :]).all()
    assert (np.diff(pos.reshape(4 * cycle, wl.n_seq), axis=0) == 1).all()
    assert ((n_end >= budgets) & (n_end <= budgets + slack)).all()


def test_bandz8k_schedule_evicts_every_call():
    wl, budgets, slack, cycle, n0 = _setup(2)
    C = wl.chunk
    pos, slots, ev, n_end = bench.window_schedule(n0, budgets, slack, C, 5)
    assert (ev == wl.n_seq).all()
    assert (slots.reshape(5, wl.n_seq, C)[:, :, 0] == budgets[None, :]).all()   # new rows from slot K each call
    assert (n_end == budgets).all()


def test_stream_bytes_and_kernel_table():
    """The algorithmic byte counts the bench divides by kernel times, on the
    32k workload's numbers, and the per-kernel table built from event records."""
    import bench
    from synth import workloads as W
    m = W.config(3).model
    row, state, band = 32 * 2 * 8 * 128 * 2, 32 * 2 * 4 * 8 * 128 * 2, 15 * 4096 * 2
    b = bench.stream_bytes(m, tokens=32 * 128, seq_calls=32, rows_moved=1000, kinds=2, one_token=False)
    assert b == {"compact_kernel": 2 * 1000 * row, "lagkv_partial_kernel": 32 * 128 * row + 32 * 2 * state}
    b = bench.stream_bytes(m, tokens=64, seq_calls=64, rows_moved=0, kinds=3, one_token=True)
    assert b["token_kernel"] == 64 * (3 * band + row + 2 * state)
    b = bench.stream_bytes(m, tokens=4, seq_calls=4, rows_moved=0, kinds=1, one_token=True)
    assert b["bandz_token_kernel"] == 4 * 3 * band and "token_kernel" not in b
    b = bench.stream_bytes(m, tokens=2048, seq_calls=1, rows_moved=0, kinds=8, one_token=False)
    assert b["lagkv_partial_kernel"] == 2048 * row              # raw variances keep no range state
    recs = [("_ZN5epikv14compact_kernelILb0EEEvv", 2.0), ("_ZN5epikv13select_kernelILb0EEEvv", 0.5),
            ("_ZN5epikv14compact_kernelILb0EEEvv", 4.0)]
    t = bench.kernel_table(recs, 2, {"compact_kernel": 6e9}, 6000.0)
    assert t["compact_kernel"]["launches_per_step"] == 1 and t["compact_kernel"]["ms_per_step"] == 3.0
    assert t["compact_kernel"]["gbs"] == pytest.approx(1000.0) and t["compact_kernel"]["hbm_frac"] == pytest.approx(1 / 6)
    assert "gbs" not in t["select_kernel"]


def test_kernel_short_names():
    from paper_2606_26472_gb300 import epikv as E
    assert E.kernel_short_name("_ZN5epikv12token_kernelILi16EEEvNS_8DevStateE") == "token_kernel"
    assert E.kernel_short_name("_ZN5epikv18bandz_token_kernelILi2EEEv") == "bandz_token_kernel"
    assert E.kernel_short_name("void epikv::compact_kernel<false, true>(epikv::DevState)") == "compact_kernel"
    assert E.kernel_short_name("_ZN5epikv20compact_stash_kernelEv") == "compact_stash_kernel"
    assert E.kernel_short_name("_ZN5epikv23compact_consumed_kernelE") == "compact_consumed_kernel"
    assert E.kernel_short_name("_ZN5epikv21select_cluster_kernelENS_8DevStateE") == "select_cluster_kernel"
    assert E.kernel_short_name("_ZN5epikv13select_kernelILb0EEEv") == "select_kernel"
    assert E.kernel_short_name("something_else") == "something_else"
