"""GPU side of the synthetic-input generator (libepikv_synth.so), producing the
same bytes as synth.gen on the device.  torch provides the device memory."""
from __future__ import annotations

import ctypes as C
import os

import numpy as np
import torch

from . import gen

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libepikv_synth.so")
_lib = None


def load():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} missing: run paper_2606_26472_gb300.build.build()")
        lib = C.CDLL(_LIB_PATH)
        lib.synth_hidden.restype = C.c_int
        lib.synth_hidden.argtypes = [C.c_uint64, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, C.c_float, C.c_float,
                                     C.c_float, C.c_float, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64,
                                     C.c_void_p]
        lib.synth_kv.restype = C.c_int
        lib.synth_kv.argtypes = [C.c_uint64, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int,
                                 C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int64,
                                 C.c_int64, C.c_int64, C.c_int64, C.c_void_p, C.c_int, C.c_int, C.c_void_p]
        lib.synth_hidden_batch.restype = C.c_int
        lib.synth_hidden_batch.argtypes = [C.c_uint64, C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_int, C.c_float,
                                           C.c_float, C.c_float, C.c_float, C.c_void_p, C.c_void_p, C.c_int64,
                                           C.c_void_p, C.c_int64, C.c_void_p]
        lib.synth_kv_batch.restype = C.c_int
        lib.synth_kv_batch.argtypes = [C.c_uint64, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_int,
                                       C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int,
                                       C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_void_p, C.c_int, C.c_int,
                                       C.c_void_p]
        lib.synth_upload_2d.restype = C.c_int
        lib.synth_upload_2d.argtypes = [C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_size_t, C.c_size_t,
                                        C.c_int, C.c_void_p]
        _lib = lib
    return _lib


def upload_2d(dst, dpitch, src, spitch, width, height, ctas, stream=None):
    """Copy of `height` rows of `width` bytes between pinned host memory and
    device memory (either direction) by SM loads and stores, no copy engine
    (see synth_upload_2d)."""
    r = load().synth_upload_2d(dst, dpitch, src, spitch, width, height, ctas, _stream(stream))
    if r != 0:
        raise RuntimeError(f"synth_upload_2d failed ({r})")


def _stream(stream):
    return (stream or torch.cuda.current_stream()).cuda_stream


class DeviceTrace:
    """Device copies of one TraceModel's tables and per-sequence segment indices."""

    def __init__(self, model: gen.TraceModel, device="cuda"):
        self.m = model
        self.tabs = gen.make_tables(model)
        self.device = device
        self.mean = torch.from_numpy(self.tabs.mean).to(device)
        self.kv_scale = torch.from_numpy(self.tabs.kv_scale).contiguous().to(device)
        self.kv_off = torch.from_numpy(self.tabs.kv_off).contiguous().to(device)
        self._seg = {}

    def seg(self, seq: int, T: int):
        t = self._seg.get(seq)
        if t is None or t.numel() < T:
            t = torch.from_numpy(gen.segment_index(self.m, seq, T)).to(self.device)
            self._seg[seq] = t
        return t

    def hidden(self, seq, layer, pos0, n, out, row_stride, stream=None):
        """Write rows of positions pos0..pos0+n-1 to `out` (a device pointer or tensor)."""
        if n <= 0:
            return
        m, tb = self.m, self.tabs
        seg = self.seg(seq, pos0 + n) if tb.seg_amp[layer] != 0 else None
        ptr = out if isinstance(out, int) else out.data_ptr()
        r = load().synth_hidden(m.seed & 0xFFFFFFFFFFFFFFFF, seq, layer, pos0, n, m.hidden, float(tb.scale[layer]),
                                float(tb.drift[layer]), float(tb.seg_amp[layer]), float(gen.INV_SD),
                                self.mean[layer].data_ptr(), seg.data_ptr() if seg is not None else None, ptr,
                                row_stride, _stream(stream))
        if r != 0:
            raise RuntimeError(f"synth_hidden failed ({r})")

    def kv(self, seq, pos0, n, slot0, k, v, *, layout, stride_layer, stride_seq=0, stride_block=0, stride_token,
           block_table=None, max_blocks=0, block_size=0, stream=None):
        """Write K and V rows of positions pos0.. to slots slot0.. of a cache view."""
        if n <= 0:
            return
        m = self.m
        r = load().synth_kv(m.seed & 0xFFFFFFFFFFFFFFFF, seq, pos0, n, slot0, m.num_layers, m.num_kv_heads,
                            m.head_dim, m.spike_per_10k, self.kv_scale.data_ptr(), self.kv_off.data_ptr(),
                            k if isinstance(k, int) else k.data_ptr(), v if isinstance(v, int) else v.data_ptr(),
                            layout, stride_layer, stride_seq, stride_block, stride_token,
                            None if block_table is None else block_table.data_ptr(), max_blocks, block_size,
                            _stream(stream))
        if r != 0:
            raise RuntimeError(f"synth_kv failed ({r})")


class DeviceBatchTrace(DeviceTrace):
    """DeviceTrace plus batched generation for ragged decode steps: every row
    of a step in one launch per layer (hidden) or one launch (K/V)."""

    def __init__(self, model, n_seq, max_len, device="cuda"):
        super().__init__(model, device)
        seg = np.stack([gen.segment_index(model, b, max_len) for b in range(n_seq)])
        self.seg_tab = torch.from_numpy(seg).to(device)
        self.seg_stride = max_len

    def hidden_batch(self, layer, seqs, pos, out, row_stride, stream=None):
        m, tb = self.m, self.tabs
        r = load().synth_hidden_batch(m.seed & 0xFFFFFFFFFFFFFFFF, layer, seqs.numel(), seqs.data_ptr(),
                                      pos.data_ptr(), m.hidden, float(tb.scale[layer]), float(tb.drift[layer]),
                                      float(tb.seg_amp[layer]), float(gen.INV_SD), self.mean[layer].data_ptr(),
                                      self.seg_tab.data_ptr(), self.seg_stride,
                                      out if isinstance(out, int) else out.data_ptr(), row_stride, _stream(stream))
        if r != 0:
            raise RuntimeError(f"synth_hidden_batch failed ({r})")

    def kv_batch(self, seqs, pos, slots, k, v, *, layout, stride_layer, stride_seq=0, stride_block=0, stride_token,
                 block_table=None, max_blocks=0, block_size=0, stream=None):
        m = self.m
        r = load().synth_kv_batch(m.seed & 0xFFFFFFFFFFFFFFFF, seqs.numel(), seqs.data_ptr(), pos.data_ptr(),
                                  slots.data_ptr(), m.num_layers, m.num_kv_heads, m.head_dim, m.spike_per_10k,
                                  self.kv_scale.data_ptr(), self.kv_off.data_ptr(),
                                  k if isinstance(k, int) else k.data_ptr(), v if isinstance(v, int) else v.data_ptr(),
                                  layout, stride_layer, stride_seq, stride_block, stride_token,
                                  None if block_table is None else block_table.data_ptr(), max_blocks, block_size,
                                  _stream(stream))
        if r != 0:
            raise RuntimeError(f"synth_kv_batch failed ({r})")


def as_u16(t: torch.Tensor) -> np.ndarray:
    """bf16 device tensor -> uint16 numpy bit patterns."""
    return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)
