"""A whole decode step (scoring, the device-side trigger, selection and the
in-place compaction) captured once in a CUDA graph and replayed step after
step from fixed staging buffers, as a serving loop would: the replays leave
the same scores, positions, lengths and cache bytes as the same steps called
one by one.  Token-level budgets and per-layer budgets."""
import numpy as np
import pytest
import torch

from paper_2606_26472_gb300 import epikv as E
from synth import workloads as W

from .harness import Session

pytestmark = pytest.mark.gpu

BANDZ, LAGKV = E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_LAGKV


def _fixed_inputs(sess, C, budgets, triggers):
    dev = sess.ws.device
    n = sess.n_seq
    seq_ids = torch.arange(n, dtype=torch.int32, device=dev)
    cu = (torch.arange(n + 1, dtype=torch.int32, device=dev) * C).contiguous()
    bud = torch.tensor(budgets, dtype=torch.int32, device=dev)
    trig = torch.tensor(triggers, dtype=torch.int32, device=dev)
    out = torch.empty((n, sess.L) if sess.layer_budgets else (n,), dtype=torch.int32, device=dev)
    hv = E.hidden_view([sess.hid[i] for i in range(sess.hid.shape[0])], sess.m.hidden)
    return seq_ids, cu, bud, trig, out, hv


@pytest.mark.parametrize("layer_budgets", [0, 1], ids=["token", "per_layer"])
def test_captured_step_replays_equal_eager_steps(gpu_lib, layer_budgets):
    model = W.small_model(71)
    C, steps = 8, 40
    kw = dict(n_seq=3, kinds=BANDZ | LAGKV, layout=E.EPIKV_LAYOUT_PAGED, max_tokens=160, max_new=C,
              prefill=(2, 0, 5), policies=(BANDZ, LAGKV, BANDZ), layer_budgets=layer_budgets)
    if layer_budgets:
        budgets = [[96, 80, 64, 48], [40, 60, 80, 100], [72, 72, 36, 36]]
        triggers = [max(k) + 7 for k in budgets]
    else:
        budgets = [96, 40, 72]
        triggers = [k + 7 for k in budgets]
    eager, graph = Session(model, **kw), Session(model, **kw)
    entries = [(b, C) for b in range(3)]
    g = None
    stream = torch.cuda.Stream()
    fixed = _fixed_inputs(graph, C, budgets, triggers)
    seq_ids, cu, bud, trig, out, hv = fixed
    for st in range(steps):
        eager.step(entries, budgets, triggers)
        graph.append(entries)              # this step's K/V and band rows, eagerly, into the fixed buffers
        torch.cuda.synchronize()
        if g is None:                      # the first step runs eagerly (first launches set up the kernels)
            E.epikv_step(graph.ctx, 3, seq_ids, cu, C, bud, trig, hv, graph.kv, out)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                E.epikv_step(graph.ctx, 3, seq_ids, cu, C, bud, trig, hv, graph.kv, out, stream=stream)
        else:
            g.replay()
        torch.cuda.synchronize()
        lens = out.cpu().numpy()
        for b in range(3):
            graph.n_seen[b] += C
            if layer_budgets:
                graph.n_layer[b] = [int(x) for x in lens[b]]
                graph.n_cache[b] = max(graph.n_layer[b])
            else:
                graph.n_cache[b] = int(lens[b])
        for b in range(3):
            assert graph.n_cache[b] == eager.n_cache[b], (st, b)
            for kind in (BANDZ, LAGKV):
                pe, se = eager.read(b, kind)
                pg, sg = graph.read(b, kind)
                np.testing.assert_array_equal(pe, pg)
                np.testing.assert_array_equal(se.view(np.uint32), sg.view(np.uint32))
            if layer_budgets:
                assert graph.n_layer[b] == eager.n_layer[b]
    for b in range(3):
        if layer_budgets:
            for l in range(model.num_layers):
                n = eager.n_layer[b][l]
                np.testing.assert_array_equal(np.stack(eager.layer_rows_u16(b, l, np.arange(n))),
                                              np.stack(graph.layer_rows_u16(b, l, np.arange(n))))
        else:
            n = eager.n_cache[b]
            np.testing.assert_array_equal(np.stack(eager.cache_rows_u16(b, np.arange(n))),
                                          np.stack(graph.cache_rows_u16(b, np.arange(n))))
    s_e, s_g = E.epikv_get_stats(eager.ctx), E.epikv_get_stats(graph.ctx)
    assert s_e == s_g and s_e["evictions"] > 3 * 10
    assert eager.error() == graph.error() == (E.EPIKV_OK, 0)
    eager.close()
    graph.close()
