"""CPU checks of the C-ABI boundary: the library builds, loads and exports
every function include/epikv.h declares, and host-side validation rejects bad
arguments before touching the GPU (no compute call is made here)."""
import ctypes as C
import os
import re

import pytest

from paper_2606_26472_gb300 import build as B
from paper_2606_26472_gb300 import epikv as E

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return E.load()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "epikv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(epikv_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert "epikv_step" in names and len(names) >= 13
    for n in names:
        assert hasattr(lib, n), n


def test_generator_library_exports(lib):
    from synth import device
    d = device.load()
    assert hasattr(d, "synth_hidden") and hasattr(d, "synth_kv")


def cfg(**kw):
    base = dict(max_seqs=4, max_cache_tokens=1024, max_new_tokens=64)
    base.update(kw)
    return E.make_config(**base)


def test_workspace_sizing_and_invalid_configs(lib):
    ok = E.epikv_workspace_bytes(cfg())
    assert ok > 0 and ok % 256 == 0
    both = E.epikv_workspace_bytes(cfg(score_kinds=3))
    assert both > ok
    # chunk-level selection adds one key per slot; 0 and 1 are the token rule
    assert E.epikv_workspace_bytes(cfg(select_chunk=0)) == E.epikv_workspace_bytes(cfg(select_chunk=1)) == ok
    assert E.epikv_workspace_bytes(cfg(select_chunk=16)) >= ok + 4 * 4 * 1024
    # per-layer budgets: per-layer lengths, masks, keep bits and kept lists
    lay = E.epikv_workspace_bytes(cfg(layer_budgets=1))
    assert lay >= ok + 4 * 1024 * (8 + 8 + 4 + 4 * 31)
    for bad in (dict(layer_budgets=2), dict(layer_budgets=1, num_layers=65),
                dict(layer_budgets=1, select_chunk=8)):
        assert E.epikv_workspace_bytes(cfg(**bad)) == 0, bad
    assert E.epikv_workspace_bytes(cfg(layer_budgets=1, num_layers=64)) > 0
    for bad in (dict(max_seqs=0), dict(head_dim=96), dict(head_dim=4), dict(hidden=4100), dict(n_band_a=0),
                dict(z_window=0), dict(score_kinds=0), dict(score_kinds=64), dict(num_kv_heads=64),
                dict(max_new_tokens=0), dict(z_window=2000), dict(score_kinds=2, lag=0),
                dict(select_chunk=-1), dict(select_chunk=65537)):
        assert E.epikv_workspace_bytes(cfg(**bad)) == 0, bad


def test_init_rejects_bad_workspace_without_gpu(lib):
    c = cfg()
    ctx = C.c_void_p()
    need = E.epikv_workspace_bytes(c)
    assert lib.epikv_init(C.byref(ctx), C.byref(c), None, need, None) == E.EPIKV_EINVAL
    assert lib.epikv_init(C.byref(ctx), C.byref(c), 0x1000 + 16, need, None) == E.EPIKV_EINVAL   # misaligned
    assert lib.epikv_init(C.byref(ctx), C.byref(c), 0x1000, need - 1, None) == E.EPIKV_EINVAL   # too small
    assert lib.epikv_init(None, C.byref(c), 0x1000, need, None) == E.EPIKV_EINVAL
    assert lib.epikv_score_update(None, 1, None, None, 1, None, None, None) == E.EPIKV_EINVAL
    assert lib.epikv_select(None, 1, None, None, None, None, 1, None, None) == E.EPIKV_EINVAL
    assert lib.epikv_compact(None, 1, None, None, 1, None, None) == E.EPIKV_EINVAL
    assert lib.epikv_step(None, 1, None, None, 1, None, None, None, None, None, None) == E.EPIKV_EINVAL
    assert E.epikv_status_string(E.EPIKV_EINVAL) == "invalid argument"
