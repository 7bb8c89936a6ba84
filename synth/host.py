"""Host-side fast path of the synthetic-input generator: the same bf16 bit
patterns as ``synth.gen.hidden_rows`` / ``synth.gen.kv_rows`` (a byte-for-byte
test pins them), produced by the plain-C twin ``libepikv_synth_host.so`` on
several host threads.  The oracle's full-size checks use it to regenerate
tens of thousands of 32-layer rows in seconds; where the library is not
built, the numpy generator is used instead (same bytes, slower)."""
from __future__ import annotations

import concurrent.futures as cf
import ctypes as C
import os

import numpy as np

from . import gen

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libepikv_synth_host.so")
_lib = None
_THREADS = max(1, min(16, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count() or 1))
_ROWS_PER_TASK = 64


def load():
    """The C generator, or None when it is not built."""
    global _lib
    if _lib is None and os.path.exists(_LIB_PATH):
        lib = C.CDLL(_LIB_PATH)
        p = C.c_void_p
        lib.synth_host_hidden.restype = C.c_int
        lib.synth_host_hidden.argtypes = [C.c_uint64, C.c_int, C.c_int, p, C.c_int64, C.c_int, C.c_float, C.c_float,
                                          C.c_float, C.c_float, p, p, p]
        lib.synth_host_kv.restype = C.c_int
        lib.synth_host_kv.argtypes = [C.c_uint64, C.c_int, C.c_int, p, p, C.c_int64, C.c_int, C.c_int, C.c_int, p, p,
                                      p]
        _lib = lib
    return _lib


def _split(n):
    return [(i, min(n, i + _ROWS_PER_TASK)) for i in range(0, n, _ROWS_PER_TASK)]


def _run_tasks(fn, n):
    parts = _split(n)
    if len(parts) <= 1 or _THREADS == 1:
        for a, b in parts:
            fn(a, b)
        return
    with cf.ThreadPoolExecutor(max_workers=_THREADS) as ex:   # the C calls release the GIL
        for f in [ex.submit(fn, a, b) for a, b in parts]:
            f.result()


def hidden_rows(m: gen.TraceModel, tabs: gen.Tables, seq: int, layer: int, positions, seg) -> np.ndarray:
    """bf16 bits [n, D]: ``gen.hidden_rows`` with the same arguments."""
    lib = load()
    if lib is None:
        return gen.hidden_rows(m, tabs, seq, layer, positions, seg)
    pos = np.ascontiguousarray(np.asarray(positions, dtype=np.int64).reshape(-1))
    n, D = pos.shape[0], m.hidden
    out = np.empty((n, D), np.uint16)
    amp = float(tabs.seg_amp[layer])
    sg = np.ascontiguousarray(np.asarray(seg)[pos].astype(np.int32)) if amp != 0 else np.zeros(n, np.int32)
    mean = np.ascontiguousarray(tabs.mean[layer], dtype=np.float32)

    def part(a, b):
        r = lib.synth_host_hidden(m.seed & 0xFFFFFFFFFFFFFFFF, seq, layer, pos[a:].ctypes.data, b - a, D,
                                  float(tabs.scale[layer]), float(tabs.drift[layer]), amp, float(gen.INV_SD),
                                  mean.ctypes.data, sg[a:].ctypes.data, out[a:].ctypes.data)
        if r != 0:
            raise RuntimeError(f"synth_host_hidden failed ({r})")

    _run_tasks(part, n)
    return out


def kv_rows(m: gen.TraceModel, tabs: gen.Tables, seq: int, kind: int, positions, spikes) -> np.ndarray:
    """bf16 bits [n, L, H, d]: ``gen.kv_rows`` with the same arguments."""
    lib = load()
    if lib is None:
        return gen.kv_rows(m, tabs, seq, kind, positions, spikes)
    pos = np.ascontiguousarray(np.asarray(positions, dtype=np.int64).reshape(-1))
    n, L, H, d = pos.shape[0], m.num_layers, m.num_kv_heads, m.head_dim
    out = np.empty((n, L, H, d), np.uint16)
    sp = np.ascontiguousarray(np.asarray(spikes)[pos].astype(np.uint8))
    scale = np.ascontiguousarray(tabs.kv_scale[kind], dtype=np.float32)
    off = np.ascontiguousarray(tabs.kv_off[kind], dtype=np.float32)

    def part(a, b):
        r = lib.synth_host_kv(m.seed & 0xFFFFFFFFFFFFFFFF, seq, kind, pos[a:].ctypes.data, sp[a:].ctypes.data, b - a,
                              L, H, d, scale.ctypes.data, off.ctypes.data, out[a:].ctypes.data)
        if r != 0:
            raise RuntimeError(f"synth_host_kv failed ({r})")

    _run_tasks(part, n)
    return out
