"""K/V pool helpers: torch-allocated bf16 pools in the layouts the library
addresses, and the epikv_kv_view that describes them."""
from __future__ import annotations

import numpy as np
import torch

from . import epikv as E


class KVCache:
    """K and V pools of L layers x H heads x d channels (bf16).

    contiguous:  k, v are [L][S][T][H][d]
    paged:       k, v are [L][num_blocks][block_size][H][d] and
                 block_table [S][max_blocks_per_seq] maps a sequence's slot
                 s to block block_table[seq][s // block_size] in every layer.
    layer_tables (paged): k, v are one pool [num_blocks][block_size][H][d]
                 and block_table [L][S][max_blocks_per_seq] gives every
                 (layer, sequence) its own blocks, so a layer that keeps
                 fewer tokens (per-layer budgets) holds fewer blocks.
    """

    def __init__(self, layout, L, H, d, *, max_seqs, max_tokens, block_size=16, num_blocks=None,
                 block_table=None, layer_tables=False, device="cuda"):
        self.layout, self.L, self.H, self.d = layout, L, H, d
        self.S, self.T = max_seqs, max_tokens
        self.block_size = block_size
        self.layer_tables = bool(layer_tables) and layout == E.EPIKV_LAYOUT_PAGED
        if layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            shape = (L, max_seqs, max_tokens, H, d)
            self.num_blocks = 0
            self.max_blocks = 0
            self.block_table = None
        else:
            self.max_blocks = (max_tokens + block_size - 1) // block_size
            per_layer = max_seqs * self.max_blocks
            if self.layer_tables:
                self.num_blocks = num_blocks if num_blocks is not None else L * per_layer
                shape = (self.num_blocks, block_size, H, d)
                if block_table is None:
                    block_table = np.arange(L * per_layer, dtype=np.int32).reshape(L, max_seqs, self.max_blocks)
            else:
                self.num_blocks = num_blocks if num_blocks is not None else per_layer
                shape = (L, self.num_blocks, block_size, H, d)
                if block_table is None:
                    block_table = np.arange(per_layer, dtype=np.int32).reshape(max_seqs, self.max_blocks)
            self.block_table = torch.as_tensor(np.asarray(block_table, dtype=np.int32)).to(device).contiguous()
        self.k = torch.empty(shape, dtype=torch.bfloat16, device=device)
        self.v = torch.empty(shape, dtype=torch.bfloat16, device=device)

    @property
    def strides(self):
        hd = self.H * self.d
        if self.layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            return dict(stride_layer=self.S * self.T * hd, stride_seq=self.T * hd, stride_block=0, stride_token=hd)
        if self.layer_tables:
            return dict(stride_layer=0, stride_seq=0, stride_block=self.block_size * hd, stride_token=hd,
                        stride_table_layer=self.S * self.max_blocks)
        return dict(stride_layer=self.num_blocks * self.block_size * hd, stride_seq=0,
                    stride_block=self.block_size * hd, stride_token=hd)

    def view(self, block_table=None):
        bt = self.block_table if block_table is None else block_table
        return E.kv_view(self.k, self.v, layout=self.layout, block_table=bt, max_blocks_per_seq=self.max_blocks,
                         block_size=self.block_size, num_blocks=self.num_blocks, **self.strides)

    def synth_kwargs(self, block_table=None):
        assert not self.layer_tables, "the generator writes one slot for every layer; use write_layer_rows"
        bt = self.block_table if block_table is None else block_table
        return dict(layout=self.layout, block_table=bt, max_blocks=self.max_blocks, block_size=self.block_size,
                    **self.strides)

    def _flat(self, layer, seq, slots, block_table_host):
        bt = block_table_host if block_table_host is not None else self.block_table.cpu().numpy()
        tab = bt[layer][seq] if self.layer_tables else bt[seq]
        return tab[slots // self.block_size] * self.block_size + slots % self.block_size

    def rows(self, kind, seq, slots, block_table_host=None):
        """bf16 rows [n, L, H, d] of the given slots (a gather on the device)."""
        pool = self.k if kind == 0 else self.v
        slots = np.asarray(slots, dtype=np.int64)
        if self.layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            idx = torch.as_tensor(slots, device=pool.device)
            return pool[:, seq].index_select(1, idx).permute(1, 0, 2, 3)
        if self.layer_tables:
            flat_pool = pool.view(-1, self.H, self.d)
            return torch.stack([flat_pool.index_select(0, torch.as_tensor(
                self._flat(l, seq, slots, block_table_host), device=pool.device)) for l in range(self.L)], dim=1)
        flat = torch.as_tensor(self._flat(0, seq, slots, block_table_host), device=pool.device)
        return pool.reshape(self.L, -1, self.H, self.d).index_select(1, flat).permute(1, 0, 2, 3)

    def write_layer_rows(self, kind, seq, layer, slots, rows, block_table_host=None):
        """Store bf16 rows [n, H, d] into the given slots of one layer (per-layer
        budgets give each layer its own slot numbering)."""
        pool = self.k if kind == 0 else self.v
        slots = np.asarray(slots, dtype=np.int64)
        if self.layout == E.EPIKV_LAYOUT_CONTIGUOUS:
            pool[layer, seq][torch.as_tensor(slots, device=pool.device)] = rows
            return
        flat = torch.as_tensor(self._flat(layer, seq, slots, block_table_host), device=pool.device)
        plane = pool.view(-1, self.H, self.d) if self.layer_tables else pool[layer].view(-1, self.H, self.d)
        plane[flat] = rows
