"""Per-token score updates captured in CUDA graphs replay to the same bits as
the same calls made one by one (each call only enqueues kernels on its
stream: no synchronisation, no allocation)."""
import numpy as np
import pytest
import torch

from paper_2606_26472_gb300 import epikv as E
from synth import gen
from synth.device import DeviceTrace

pytestmark = pytest.mark.gpu


def _setup(m, B, T):
    cfg = E.make_config(max_seqs=B, max_cache_tokens=T, max_new_tokens=1, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), score_kinds=E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_HSVAR)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device="cuda")
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(B):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_BANDZ)
    return ctx, ws


def test_graph_replay_equals_eager_per_token_updates(gpu_lib):
    m = gen.TraceModel(0xE91C0004)
    B, T, G = 4, 320, 64
    dt = DeviceTrace(m)
    nb = len(m.band_layers)
    hid = torch.empty((nb, T, B, m.hidden), dtype=torch.bfloat16, device="cuda")
    for i, layer in enumerate(m.band_layers):
        for b in range(B):
            dt.hidden(b, layer, 0, T, hid[i, :, b].data_ptr(), B * m.hidden)
    seq_ids = torch.arange(B, dtype=torch.int32, device="cuda")
    cu = torch.arange(B + 1, dtype=torch.int32, device="cuda")
    step_bytes = B * m.hidden * 2
    bases = [hid[i].data_ptr() for i in range(nb)]

    def view(t):
        hv = E.epikv_hidden_view()
        hv.row_stride = m.hidden
        for i in range(nb):
            hv.band_rows[i] = bases[i] + t * step_bytes
        return hv

    kv_dummy = E.kv_view(hid, hid, stride_layer=0, stride_seq=0, stride_token=8 * 128)   # not read by band kinds

    # eager: one call per token
    ctx_e, ws_e = _setup(m, B, T)
    for t in range(T):
        E.epikv_score_update(ctx_e, B, seq_ids, cu, 1, view(t), kv_dummy)
    # graphs: the first token eagerly (first launches size the grids), then
    # the rest in graphs of G tokens
    ctx_g, ws_g = _setup(m, B, T)
    E.epikv_score_update(ctx_g, B, seq_ids, cu, 1, view(0), kv_dummy)
    torch.cuda.synchronize()
    t = 1
    graphs = []
    while t < T:
        n = min(G, T - t)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for k in range(n):
                E.epikv_score_update(ctx_g, B, seq_ids, cu, 1, view(t + k), kv_dummy)
        graphs.append(g)
        t += n
    for g in graphs:
        g.replay()
    torch.cuda.synchronize()
    for b in range(B):
        for kind in (E.EPIKV_SCORE_BANDZ, E.EPIKV_SCORE_HSVAR):
            pe, se, ne = E.epikv_read_slots(ctx_e, b, kind, T)
            pg, sg, ng = E.epikv_read_slots(ctx_g, b, kind, T)
            assert ne == ng == T
            np.testing.assert_array_equal(pe, pg)
            np.testing.assert_array_equal(np.array(se, np.float32), np.array(sg, np.float32))
    assert E.epikv_get_error(ctx_g) == (E.EPIKV_OK, 0)
