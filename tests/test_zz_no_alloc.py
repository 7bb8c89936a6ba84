"""The allocation-free Lag-KV entry point against the context path and the
fp64 oracle.

epikv_lagkv_score_noalloc serves callers that cannot allocate device memory
(no workspace, no context): its scratch is a fixed array inside the library.
This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes alone in a fresh process.
"""
import ctypes as C

import numpy as np
import pytest
import torch

from paper_2606_26472_gb300 import epikv as E
from paper_2606_26472_gb300.cache import KVCache
from synth import gen
from synth.device import DeviceTrace

from .harness import OracleTrace, assert_scores_close

pytestmark = pytest.mark.gpu

SCRATCH_FLOATS = 1 << 19


def test_noalloc_scores_match_the_context_path_on_two_calls(gpu_lib):
    lib = gpu_lib
    model = gen.TraceModel(0xE91C0003)
    L, H, d = model.num_layers, model.num_kv_heads, model.head_dim
    lens = (1500, 700)
    T = 1536
    bt = gen.block_permutation(9, 2 * (T // 16)).reshape(2, T // 16)
    cache = KVCache(E.EPIKV_LAYOUT_PAGED, L, H, d, max_seqs=2, max_tokens=T, block_table=bt)
    dt = DeviceTrace(model)
    for b, n in enumerate(lens):
        dt.kv(b, 0, n, 0, cache.k, cache.v, **cache.synth_kwargs())
    view = cache.view()

    # the existing entry point: a context fed in decode chunks
    cfg = E.make_config(max_seqs=2, max_cache_tokens=T, max_new_tokens=256, num_layers=L, num_kv_heads=H,
                        head_dim=d, lag=16, lag_window=64, score_kinds=E.EPIKV_SCORE_LAGKV)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device="cuda")
    ctx = E.epikv_init(cfg, ws, ws.numel())
    ref = []
    for b, n in enumerate(lens):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_LAGKV)
        done = 0
        while done < n:
            c = min(256, n - done)
            ids = torch.tensor([b], dtype=torch.int32, device="cuda")
            cu = torch.tensor([0, c], dtype=torch.int32, device="cuda")
            E.epikv_score_update(ctx, 1, ids, cu, c, None, view)
            done += c
        _, sc, m = E.epikv_read_slots(ctx, b, E.EPIKV_SCORE_LAGKV, T)
        assert m == n
        ref.append(np.array(sc, dtype=np.float32))
    assert E.epikv_get_error(ctx) == (E.EPIKV_OK, 0)
    E.epikv_destroy(ctx)

    # the new entry point through the C ABI, two calls in a row on one stream
    out = torch.full((2, T), float("nan"), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    for b, n in enumerate(lens):
        st = lib.epikv_lagkv_score_noalloc(C.byref(view), b, n, L, H, d, 16, C.c_float(1e-6), 64,
                                           out[b].data_ptr(), stream)
        assert st == E.EPIKV_OK
    torch.cuda.synchronize()
    for b, n in enumerate(lens):
        got = out[b, :n].cpu().numpy()
        assert_scores_close(got, ref[b], f"no-alloc seq {b}")
        assert np.all(np.isnan(out[b, n:].cpu().numpy()))   # nothing written past n
    # and both against the fp64 oracle, position by position
    orc = OracleTrace(model, dt.tabs, 1, lens[1], E.EPIKV_SCORE_LAGKV)
    assert_scores_close(out[1, :lens[1]].cpu().numpy(), orc.scores[E.EPIKV_SCORE_LAGKV], "no-alloc vs oracle")

    # a request larger than the fixed scratch is refused before any launch
    too_many = SCRATCH_FLOATS // (2 * L) + 1
    st = lib.epikv_lagkv_score_noalloc(C.byref(view), 0, too_many, L, H, d, 16, C.c_float(1e-6), 64,
                                       out[0].data_ptr(), stream)
    assert st == E.EPIKV_EINVAL


# head shapes at the edges of what the entry point accepts, both layouts, a
# one-token window, a window that does not divide the tile, the largest
# window, and lags that do not divide n
SHAPES = [
    ("d8_h32_paged_w1_lag5", 32, 8, E.EPIKV_LAYOUT_PAGED, 1, 5, 301),
    ("d64_h4_contig_w200_lag16", 4, 64, E.EPIKV_LAYOUT_CONTIGUOUS, 200, 16, 517),
    ("d256_h8_paged_w1024_lag7", 8, 256, E.EPIKV_LAYOUT_PAGED, 1024, 7, 1100),
    ("d128_h8_contig_w64_lag16", 8, 128, E.EPIKV_LAYOUT_CONTIGUOUS, 64, 16, 777),
]


@pytest.mark.parametrize("name,H,d,layout,window,lag,n", SHAPES, ids=[c[0] for c in SHAPES])
def test_noalloc_matches_the_oracle(gpu_lib, name, H, d, layout, window, lag, n):
    lib = gpu_lib
    model = gen.TraceModel(0xE91C0200 + H * d + window, num_layers=3, hidden=256, num_kv_heads=H, head_dim=d,
                           band_a=(1,), band_b=(2,))
    L = model.num_layers
    T = (n + 15) // 16 * 16 + 16
    seqs = 2
    bt = gen.block_permutation(31, seqs * (T // 16)).reshape(seqs, T // 16) if layout else None
    cache = KVCache(layout, L, H, d, max_seqs=seqs, max_tokens=T, block_table=bt)
    dt = DeviceTrace(model)
    dt.kv(1, 0, n, 0, cache.k, cache.v, **cache.synth_kwargs())
    view = cache.view()
    out = torch.full((2, T), float("nan"), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    for rep in range(2):       # two calls in a row: the second finds the first's scratch contents
        st = lib.epikv_lagkv_score_noalloc(C.byref(view), 1, n, L, H, d, lag, C.c_float(1e-6), window,
                                           out[rep].data_ptr(), stream)
        assert st == E.EPIKV_OK
    torch.cuda.synchronize()
    ref = OracleTrace(model, dt.tabs, 1, n, E.EPIKV_SCORE_LAGKV, lag=lag, lag_window=window)
    for rep in range(2):
        assert_scores_close(out[rep, :n].cpu().numpy(), ref.scores[E.EPIKV_SCORE_LAGKV], f"{name} call {rep}")
        assert np.all(np.isnan(out[rep, n:].cpu().numpy()))
