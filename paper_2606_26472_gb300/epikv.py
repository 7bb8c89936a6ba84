"""Thin ctypes binding of libepikv (include/epikv.h): the same names, argument
marshalling only.  Every step of the eviction path runs in the library's CUDA
kernels; there is no Python or CPU fallback, and loading fails loudly when the
library is missing."""
from __future__ import annotations

import ctypes as C
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libepikv.so")

EPIKV_OK, EPIKV_EINVAL, EPIKV_ECUDA, EPIKV_EDEVICE = 0, 1, 2, 3
EPIKV_DEV_OK, EPIKV_DEV_BATCH, EPIKV_DEV_CAPACITY, EPIKV_DEV_SLOT = 0, 1, 2, 3
EPIKV_DEV_KEPT, EPIKV_DEV_BUDGET, EPIKV_DEV_TIMEOUT = 4, 5, 6
EPIKV_SCORE_BANDZ, EPIKV_SCORE_LAGKV, EPIKV_SCORE_HSVAR = 1, 2, 4
EPIKV_SCORE_KVKEY, EPIKV_SCORE_KVVAL, EPIKV_SCORE_LAGKEY = 8, 16, 32
EPIKV_LAYOUT_CONTIGUOUS, EPIKV_LAYOUT_PAGED = 0, 1


class epikv_config(C.Structure):
    _fields_ = [("max_seqs", C.c_int32), ("max_cache_tokens", C.c_int32), ("max_new_tokens", C.c_int32),
                ("num_layers", C.c_int32), ("num_kv_heads", C.c_int32), ("head_dim", C.c_int32),
                ("hidden", C.c_int32), ("n_band_a", C.c_int32), ("n_band_b", C.c_int32),
                ("z_window", C.c_int32), ("z_eps", C.c_float), ("lag", C.c_int32), ("lag_eps", C.c_float),
                ("lag_window", C.c_int32), ("recency_cap", C.c_int32), ("score_kinds", C.c_int32),
                ("select_chunk", C.c_int32), ("layer_budgets", C.c_int32)]


class epikv_hidden_view(C.Structure):
    _fields_ = [("band_rows", C.c_void_p * 32), ("row_stride", C.c_int64)]


class epikv_kv_view(C.Structure):
    _fields_ = [("k", C.c_void_p), ("v", C.c_void_p), ("layout", C.c_int32), ("stride_layer", C.c_int64),
                ("stride_seq", C.c_int64), ("stride_block", C.c_int64), ("stride_token", C.c_int64),
                ("block_table", C.c_void_p), ("max_blocks_per_seq", C.c_int32), ("block_size", C.c_int32),
                ("num_blocks", C.c_int32), ("stride_table_layer", C.c_int64)]


class epikv_stats(C.Structure):
    _fields_ = [("tokens_scored", C.c_ulonglong), ("evictions", C.c_ulonglong), ("rows_moved", C.c_ulonglong),
                ("layer_rows_moved", C.c_ulonglong)]


_P = C.c_void_p
_I = C.c_int32
_SIGS = {
    "epikv_workspace_bytes": (C.c_size_t, [C.POINTER(epikv_config)]),
    "epikv_init": (C.c_int, [C.POINTER(_P), C.POINTER(epikv_config), _P, C.c_size_t, _P]),
    "epikv_seq_reset": (C.c_int, [_P, _I, _I, _I, _P]),
    "epikv_score_update": (C.c_int, [_P, _I, _P, _P, _I, C.POINTER(epikv_hidden_view),
                                     C.POINTER(epikv_kv_view), _P]),
    "epikv_select": (C.c_int, [_P, _I, _P, _P, _P, _P, _I, _P, _P]),
    "epikv_compact": (C.c_int, [_P, _I, _P, _P, _I, C.POINTER(epikv_kv_view), _P]),
    "epikv_step": (C.c_int, [_P, _I, _P, _P, _I, _P, _P, C.POINTER(epikv_hidden_view),
                             C.POINTER(epikv_kv_view), _P, _P]),
    "epikv_set_phase_events": (C.c_int, [_P, _P]),
    "epikv_set_kernel_events": (C.c_int, [_P, _P, _I, _P, C.POINTER(_I)]),
    "epikv_read_slots": (C.c_int, [_P, _I, _I, _P, _P, _I, C.POINTER(_I)]),
    "epikv_read_layer_slots": (C.c_int, [_P, _I, _I, _P, _I, C.POINTER(_I)]),
    "epikv_get_stats": (C.c_int, [_P, C.POINTER(epikv_stats)]),
    "epikv_get_error": (C.c_int, [_P, C.POINTER(_I)]),
    "epikv_lagkv_score_noalloc": (C.c_int, [C.POINTER(epikv_kv_view), _I, _I, _I, _I, _I, _I, C.c_float, _I,
                                            _P, _P]),
    "epikv_destroy": (None, [_P]),
    "epikv_status_string": (C.c_char_p, [C.c_int]),
}

_lib = None


def load(path: str = LIB_PATH):
    """Load libepikv.so (built in-tree by paper_2606_26472_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"libepikv.so not found at {path}: run paper_2606_26472_gb300.build.build() first "
                           "(the eviction path has no fallback)")
    lib = C.CDLL(path)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


class EpikvError(RuntimeError):
    def __init__(self, status, what):
        msg = load().epikv_status_string(status).decode()
        super().__init__(f"{what}: {msg} (status {status})")
        self.status = status


def _check(status, what):
    if status != EPIKV_OK:
        raise EpikvError(status, what)


def _ptr(x):
    """Device/host pointer of a torch tensor, an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return s if isinstance(s, int) else s.cuda_stream


def make_config(*, max_seqs, max_cache_tokens, max_new_tokens, num_layers=32, num_kv_heads=8, head_dim=128,
                hidden=4096, n_band_a=7, n_band_b=8, z_window=64, z_eps=1e-6, lag=16, lag_eps=1e-6,
                lag_window=64, recency_cap=128, score_kinds=EPIKV_SCORE_BANDZ, select_chunk=1, layer_budgets=0):
    return epikv_config(max_seqs, max_cache_tokens, max_new_tokens, num_layers, num_kv_heads, head_dim, hidden,
                        n_band_a, n_band_b, z_window, z_eps, lag, lag_eps, lag_window, recency_cap, score_kinds,
                        select_chunk, layer_budgets)


def hidden_view(band_rows, row_stride):
    hv = epikv_hidden_view()
    for i, r in enumerate(band_rows):
        hv.band_rows[i] = _ptr(r)
    hv.row_stride = row_stride
    return hv


def kv_view(k, v, *, layout=EPIKV_LAYOUT_CONTIGUOUS, stride_layer, stride_seq=0, stride_block=0, stride_token,
            block_table=None, max_blocks_per_seq=0, block_size=0, num_blocks=0, stride_table_layer=0):
    return epikv_kv_view(_ptr(k), _ptr(v), layout, stride_layer, stride_seq, stride_block, stride_token,
                         _ptr(block_table), max_blocks_per_seq, block_size, num_blocks, stride_table_layer)


# ---------------------------------------------------------------- same names
def epikv_workspace_bytes(cfg):
    return load().epikv_workspace_bytes(C.byref(cfg))


def epikv_init(cfg, workspace, workspace_bytes, stream=None):
    ctx = C.c_void_p()
    _check(load().epikv_init(C.byref(ctx), C.byref(cfg), _ptr(workspace), workspace_bytes, _stream(stream)),
           "epikv_init")
    return ctx


def epikv_seq_reset(ctx, seq, prefill_len=0, policy=EPIKV_SCORE_BANDZ, stream=None):
    _check(load().epikv_seq_reset(ctx, seq, prefill_len, policy, _stream(stream)), "epikv_seq_reset")


def epikv_score_update(ctx, n_seq, seq_ids, cu_new, max_new, hidden, kv, stream=None):
    _check(load().epikv_score_update(ctx, n_seq, _ptr(seq_ids), _ptr(cu_new), max_new,
                                     C.byref(hidden) if hidden is not None else None,
                                     C.byref(kv) if kv is not None else None, _stream(stream)),
           "epikv_score_update")


def epikv_select(ctx, n_seq, seq_ids, budget, trigger, kept, kept_stride, n_kept, stream=None):
    _check(load().epikv_select(ctx, n_seq, _ptr(seq_ids), _ptr(budget), _ptr(trigger), _ptr(kept), kept_stride,
                               _ptr(n_kept), _stream(stream)), "epikv_select")


def epikv_compact(ctx, n_seq, seq_ids, kept, kept_stride, kv, stream=None):
    _check(load().epikv_compact(ctx, n_seq, _ptr(seq_ids), _ptr(kept), kept_stride, C.byref(kv), _stream(stream)),
           "epikv_compact")


def epikv_step(ctx, n_seq, seq_ids, cu_new, max_new, budget, trigger, hidden, kv, n_cache_out=None, stream=None):
    _check(load().epikv_step(ctx, n_seq, _ptr(seq_ids), _ptr(cu_new), max_new, _ptr(budget), _ptr(trigger),
                             C.byref(hidden) if hidden is not None else None, C.byref(kv), _ptr(n_cache_out),
                             _stream(stream)),
           "epikv_step")


def epikv_set_phase_events(ctx, events):
    """events: four torch.cuda.Event(enable_timing=True) or None."""
    if events is None:
        _check(load().epikv_set_phase_events(ctx, None), "epikv_set_phase_events")
        return
    arr = (C.c_void_p * 4)(*[e.cuda_event for e in events])
    _check(load().epikv_set_phase_events(ctx, arr), "epikv_set_phase_events")


class KernelClock:
    """Per-kernel CUDA events of a context (epikv_set_kernel_events): every
    kernel the context's calls launch is bracketed by two events on its
    stream.  `start()` arms it, `stop()` returns [(kernel name, ms)] in launch
    order (synchronising on the last event)."""

    def __init__(self, ctx, cap):
        import torch
        self.ctx, self.cap = ctx, cap
        self.events = [torch.cuda.Event(enable_timing=True) for _ in range(2 * cap)]
        s = torch.cuda.current_stream()
        for e in self.events:
            e.record(s)            # materialise the handles
        self._ev = (C.c_void_p * (2 * cap))(*[e.cuda_event for e in self.events])
        self._names = (C.c_char_p * cap)()

    def start(self):
        _check(load().epikv_set_kernel_events(self.ctx, self._ev, self.cap, self._names, None),
               "epikv_set_kernel_events")

    def stop(self):
        used = C.c_int32()
        _check(load().epikv_set_kernel_events(self.ctx, None, 0, None, C.byref(used)), "epikv_set_kernel_events")
        n = used.value
        if n:
            self.events[2 * n - 1].synchronize()
        return [((self._names[k] or b"?").decode(), self.events[2 * k].elapsed_time(self.events[2 * k + 1]))
                for k in range(n)]


def kernel_short_name(name):
    """'epikv::compact_kernel<true>' style names from the runtime's (possibly
    mangled) kernel name: the function's identifier only."""
    import re
    for ident in ("bandz_g_kernel", "bandz_token_kernel", "lagkv_partial_kernel", "score_finalize_kernel",
                  "token_kernel", "select_cluster_kernel", "select_kernel", "layer_keep_kernel", "layer_union_kernel", "compact_stash_kernel",
                  "compact_consumed_kernel", "compact_kernel"):
        if re.search(r"(?<![A-Za-z_])" + ident, name):
            return ident
    return name


def epikv_read_slots(ctx, seq, kind, cap):
    """Synchronising read-back: (positions, scores of `kind`) as lists."""
    n = C.c_int32()
    score = (C.c_float * max(cap, 1))()
    pos = (C.c_int32 * max(cap, 1))()
    _check(load().epikv_read_slots(ctx, seq, kind, score, pos, cap, C.byref(n)), "epikv_read_slots")
    m = min(n.value, cap)
    return list(pos[:m]), list(score[:m]), n.value


def epikv_read_layer_slots(ctx, seq, layer, cap):
    """Synchronising read-back under per-layer budgets: (positions of the
    layer's slots as a list, the layer's length)."""
    n = C.c_int32()
    pos = (C.c_int32 * max(cap, 1))()
    _check(load().epikv_read_layer_slots(ctx, seq, layer, pos, cap, C.byref(n)), "epikv_read_layer_slots")
    return list(pos[:min(n.value, cap)]), n.value


def epikv_get_stats(ctx):
    s = epikv_stats()
    _check(load().epikv_get_stats(ctx, C.byref(s)), "epikv_get_stats")
    return {"tokens_scored": s.tokens_scored, "evictions": s.evictions, "rows_moved": s.rows_moved,
            "layer_rows_moved": s.layer_rows_moved}


def epikv_get_error(ctx):
    """(status, device code); clears the sticky device error word."""
    code = C.c_int32()
    st = load().epikv_get_error(ctx, C.byref(code))
    return st, code.value


def epikv_lagkv_score_noalloc(kv, seq, n, num_layers, num_kv_heads, head_dim, lag, lag_eps, window, scores,
                              stream=None):
    """Lag-KV scores of positions 0..n-1 of `seq` without any workspace (see epikv.h)."""
    _check(load().epikv_lagkv_score_noalloc(C.byref(kv), seq, n, num_layers, num_kv_heads, head_dim, lag, lag_eps,
                                            window, _ptr(scores), _stream(stream)), "epikv_lagkv_score_noalloc")


def epikv_destroy(ctx):
    load().epikv_destroy(ctx)


def epikv_status_string(status):
    return load().epikv_status_string(status).decode()
