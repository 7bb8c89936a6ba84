"""K/V pool helpers: torch-allocated bf16 pools in the two layouts the library
addresses, and the epikv_kv_view that describes them."""
from __future__ import annotations

import numpy as np
import torch

from . import epikv as E


class KVCache:
    """K and V pools of L layers x H heads x d channels (bf16).

    contiguous: k, v are [L][S][T][H][d]
    paged:      k, v are [L][num_blocks][block_size][H][d] and
                block_table [S][max_blocks_per_seq] maps a sequence's slot
                s to block block_table[seq][s // block_size].
    """

    def __init__(self, layout, L, H, d, *, max_seqs, max_tokens, block_size=16, num_blocks=None,
                 block_table=None, device="cuda"):
        self.layout, self.L, self.H, self.d = layout, L, H, d
        self.S, self.T = max_seqs, max_tokens
        self.block_size = block_size
        if layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            shape = (L, max_seqs, max_tokens, H, d)
            self.num_blocks = 0
            self.max_blocks = 0
            self.block_table = None
        else:
            self.max_blocks = (max_tokens + block_size - 1) // block_size
            self.num_blocks = num_blocks if num_blocks is not None else max_seqs * self.max_blocks
            shape = (L, self.num_blocks, block_size, H, d)
            if block_table is None:
                block_table = np.arange(max_seqs * self.max_blocks, dtype=np.int32).reshape(max_seqs, self.max_blocks)
            self.block_table = torch.as_tensor(np.asarray(block_table, dtype=np.int32)).to(device).contiguous()
        self.k = torch.empty(shape, dtype=torch.bfloat16, device=device)
        self.v = torch.empty(shape, dtype=torch.bfloat16, device=device)

    @property
    def strides(self):
        hd = self.H * self.d
        if self.layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            return dict(stride_layer=self.S * self.T * hd, stride_seq=self.T * hd, stride_block=0, stride_token=hd)
        return dict(stride_layer=self.num_blocks * self.block_size * hd, stride_seq=0,
                    stride_block=self.block_size * hd, stride_token=hd)

    def view(self, block_table=None):
        bt = self.block_table if block_table is None else block_table
        return E.kv_view(self.k, self.v, layout=self.layout, block_table=bt, max_blocks_per_seq=self.max_blocks,
                         block_size=self.block_size, num_blocks=self.num_blocks, **self.strides)

    def synth_kwargs(self, block_table=None):
        bt = self.block_table if block_table is None else block_table
        return dict(layout=self.layout, block_table=bt, max_blocks=self.max_blocks, block_size=self.block_size,
                    **self.strides)

    def rows(self, kind, seq, slots, block_table_host=None):
        """bf16 rows [n, L, H, d] of the given slots (a gather on the device)."""
        pool = self.k if kind == 0 else self.v
        slots = np.asarray(slots, dtype=np.int64)
        if self.layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            idx = torch.as_tensor(slots, device=pool.device)
            return pool[:, seq].index_select(1, idx).permute(1, 0, 2, 3)
        bt = block_table_host if block_table_host is not None else self.block_table.cpu().numpy()
        blk = bt[seq][slots // self.block_size]
        off = slots % self.block_size
        flat = torch.as_tensor(blk * self.block_size + off, device=pool.device)
        return pool.reshape(self.L, -1, self.H, self.d).index_select(1, flat).permute(1, 0, 2, 3)

    def write_layer_rows(self, kind, seq, layer, slots, rows, block_table_host=None):
        """Store bf16 rows [n, H, d] into the given slots of one layer (per-layer
        budgets give each layer its own slot numbering)."""
        pool = self.k if kind == 0 else self.v
        slots = np.asarray(slots, dtype=np.int64)
        if self.layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            pool[layer, seq][torch.as_tensor(slots, device=pool.device)] = rows
            return
        bt = block_table_host if block_table_host is not None else self.block_table.cpu().numpy()
        flat = bt[seq][slots // self.block_size] * self.block_size + slots % self.block_size
        pool[layer].view(-1, self.H, self.d)[torch.as_tensor(flat, device=pool.device)] = rows
