"""Host logic of bench.py's decode-window workloads (no GPU): the ragged
64-sequence schedule evicts every sequence exactly once per 65 calls, one
sequence per call but one, and never writes past a cache's capacity; the
8 x 8k schedule evicts every sequence at every call."""
import numpy as np

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
