"""Decode-loop integration: a LLaMA-shaped, random-weight model driving EpiKV.

The model's own forward pass produces everything the eviction path reads:
the per-layer hidden states (the output_hidden_states rows of the Band A and
Band B layers) and the post-RoPE keys and values, written into a paged KV
pool at each sequence's next cache slot.  After every token the decode loop
calls epikv_step, which scores the token, and, when a sequence's cache passes
its trigger, selects the kept tokens and compacts every layer's K/V in place;
attention then runs over exactly the kept tokens.  Nothing in the model is
changed for eviction: the cache it attends over is simply shorter.

The weights are random (no checkpoint is available), so the tokens carry no
meaning and there is no accuracy claim; the demo checks the plumbing.

    python examples/llama_decode.py --layers 32 --hidden 4096 --steps 256
"""
from __future__ import annotations

import argparse
import dataclasses
import math
import os
import sys

import numpy as np
import torch
import torch.nn.functional as F

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2606_26472_gb300 import epikv as E  # noqa: E402
from paper_2606_26472_gb300.cache import KVCache  # noqa: E402


@dataclasses.dataclass
class ModelShape:
    layers: int = 32
    hidden: int = 4096
    heads: int = 32
    kv_heads: int = 8
    head_dim: int = 128
    mlp: int = 14336
    vocab: int = 32000
    band_a: tuple = tuple(range(7, 14))
    band_b: tuple = tuple(range(18, 26))


def small_shape():
    return ModelShape(layers=8, hidden=512, heads=8, kv_heads=2, head_dim=64, mlp=1024, vocab=1000,
                      band_a=(2, 3), band_b=(5, 6))


class RandomLlama:
    """A decoder-only transformer with the LLaMA block (RMSNorm, RoPE, GQA
    attention, SwiGLU MLP) and random bf16 weights."""

    def __init__(self, shape: ModelShape, seed: int = 0, device="cuda"):
        self.s = shape
        g = torch.Generator(device=device).manual_seed(seed)
        bf = torch.bfloat16

        def w(n_in, n_out):
            return (torch.randn(n_in, n_out, generator=g, device=device) / math.sqrt(n_in)).to(bf)

        s = shape
        self.embed = torch.randn(s.vocab, s.hidden, generator=g, device=device).to(bf)
        self.layers = []
        for _ in range(s.layers):
            self.layers.append(dict(wq=w(s.hidden, s.heads * s.head_dim), wk=w(s.hidden, s.kv_heads * s.head_dim),
                                    wv=w(s.hidden, s.kv_heads * s.head_dim), wo=w(s.heads * s.head_dim, s.hidden),
                                    w1=w(s.hidden, s.mlp), w3=w(s.hidden, s.mlp), w2=w(s.mlp, s.hidden)))
        self.lm_head = w(s.hidden, s.vocab)
        inv = 1.0 / (10000.0 ** (torch.arange(0, s.head_dim, 2, device=device, dtype=torch.float32) / s.head_dim))
        self.inv_freq = inv

    @staticmethod
    def _rms(x):
        xf = x.float()
        return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + 1e-5)).to(x.dtype)

    def _rope(self, x, pos):
        # x [B, n, d], pos [B]
        ang = pos.float()[:, None] * self.inv_freq[None, :]             # [B, d/2]
        cos, sin = ang.cos()[:, None, :], ang.sin()[:, None, :]
        x1, x2 = x.float()[..., 0::2], x.float()[..., 1::2]
        out = torch.stack([x1 * cos - x2 * sin, x1 * sin + x2 * cos], dim=-1).flatten(-2)
        return out.to(x.dtype)

    def step(self, tokens, positions, cache: KVCache, seqs, slots, lengths):
        """One decode token per sequence.  K/V of the new tokens are written at
        `slots`; attention spans slots [0, lengths).  Returns (logits, the
        hidden state after every layer [layers][B, hidden])."""
        s = self.s
        B = tokens.shape[0]
        x = self.embed[tokens]
        hs = []
        bs = cache.block_size
        bt = cache.block_table[seqs]                                      # [B, max_blocks]
        max_len = int(lengths.max())
        j = torch.arange(max_len, device=x.device)
        blk = bt.gather(1, (j // bs)[None, :].expand(B, -1).clamp(max=bt.shape[1] - 1))
        flat = blk * bs + (j % bs)[None, :]                              # [B, max_len] pool rows
        mask = j[None, :] < lengths[:, None]
        new_flat = bt.gather(1, (slots // bs)[:, None])[:, 0] * bs + slots % bs
        for l, p in enumerate(self.layers):
            h = self._rms(x)
            q = (h @ p["wq"]).view(B, s.heads, s.head_dim)
            k = (h @ p["wk"]).view(B, s.kv_heads, s.head_dim)
            v = (h @ p["wv"]).view(B, s.kv_heads, s.head_dim)
            q = self._rope(q, positions)
            k = self._rope(k, positions)
            kp = cache.k[l].view(-1, s.kv_heads, s.head_dim)
            vp = cache.v[l].view(-1, s.kv_heads, s.head_dim)
            kp[new_flat] = k
            vp[new_flat] = v
            K = kp[flat].transpose(1, 2)                                 # [B, kvh, len, d]
            V = vp[flat].transpose(1, 2)
            rep = s.heads // s.kv_heads
            K = K.repeat_interleave(rep, dim=1)
            V = V.repeat_interleave(rep, dim=1)
            o = F.scaled_dot_product_attention(q[:, :, None, :], K, V, attn_mask=mask[:, None, None, :])
            x = x + o.reshape(B, s.heads * s.head_dim) @ p["wo"]
            h2 = self._rms(x)
            x = x + (F.silu(h2 @ p["w1"]) * (h2 @ p["w3"])) @ p["w2"]
            hs.append(x)
        return self._rms(x) @ self.lm_head, hs


@dataclasses.dataclass
class DecodeResult:
    tokens: np.ndarray           # [B, steps]
    n_cache: list
    evictions: int
    band_rows: dict              # (seq, layer) -> uint16 [T, hidden] (recorded when asked)
    kv_rows: dict                # seq -> (K, V) uint16 [T, L, H, d]
    ctx: object
    cache: KVCache


def decode(shape: ModelShape, *, batch=4, prompt=8, steps=200, budget=96, slack=16, seed=0, record=False,
           kinds=E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_LAGKV, device="cuda"):
    """Greedy decode of `batch` random prompts for `steps` tokens with EpiKV
    eviction (budget K, evict when the cache passes K + slack)."""
    model = RandomLlama(shape, seed, device)
    s = shape
    T_cap = budget + slack + 1
    bands = list(shape.band_a) + list(shape.band_b)
    mb = (T_cap + 15) // 16
    perm = torch.randperm(batch * mb, generator=torch.Generator().manual_seed(seed)).numpy().reshape(batch, mb)
    cache = KVCache(E.EPIKV_LAYOUT_PAGED, s.layers, s.kv_heads, s.head_dim, max_seqs=batch, max_tokens=T_cap,
                    block_table=perm, device=device)
    cfg = E.make_config(max_seqs=batch, max_cache_tokens=T_cap, max_new_tokens=1, num_layers=s.layers,
                        num_kv_heads=s.kv_heads, head_dim=s.head_dim, hidden=s.hidden,
                        n_band_a=len(shape.band_a), n_band_b=len(shape.band_b), score_kinds=kinds)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device=device)
    ctx = E.epikv_init(cfg, ws, ws.numel())
    policies = [E.EPIKV_SCORE_BANDZ if b % 2 == 0 or not kinds & E.EPIKV_SCORE_LAGKV else E.EPIKV_SCORE_LAGKV
                for b in range(batch)]
    for b in range(batch):
        E.epikv_seq_reset(ctx, b, prompt, policies[b])
    g = torch.Generator(device=device).manual_seed(seed + 1)
    prompts = torch.randint(0, s.vocab, (batch, prompt), generator=g, device=device)
    seqs = torch.arange(batch, device=device)
    seq_ids = seqs.to(torch.int32)
    cu = torch.arange(batch + 1, dtype=torch.int32, device=device)
    bud = torch.full((batch,), budget, dtype=torch.int32, device=device)
    trig = bud + slack
    n_out = torch.empty(batch, dtype=torch.int32, device=device)
    n_cache = torch.zeros(batch, dtype=torch.int64, device=device)
    out_tokens = []
    band_rows = {}
    kv_rows = {b: ([], []) for b in range(batch)}
    evictions = 0
    tok = prompts[:, 0]
    total = prompt + steps
    for t in range(total):
        pos = torch.full((batch,), t, dtype=torch.int64, device=device)
        slots = n_cache.clone()
        logits, hs = model.step(tok, pos, cache, seqs, slots, n_cache + 1)
        rows = [hs[l].contiguous() for l in bands]
        hv = E.hidden_view(rows, s.hidden)
        if record:
            for b in range(batch):
                for l, r in zip(bands, rows):
                    band_rows.setdefault((b, l), []).append(r[b].view(torch.int16).cpu().numpy().view(np.uint16))
                blk = cache.block_table[b, int(slots[b]) // 16].item() * 16 + int(slots[b]) % 16
                kv_rows[b][0].append(cache.k[:, blk // 16, blk % 16].view(torch.int16).cpu().numpy().view(np.uint16))
                kv_rows[b][1].append(cache.v[:, blk // 16, blk % 16].view(torch.int16).cpu().numpy().view(np.uint16))
        E.epikv_step(ctx, batch, seq_ids, cu, 1, bud, trig, hv, cache.view(), n_out)
        new_len = n_out.to(torch.int64)
        evictions += int((new_len < n_cache + 1).sum())
        n_cache = new_len
        tok = prompts[:, t + 1] if t + 1 < prompt else logits.argmax(-1)
        if t >= prompt:
            out_tokens.append(tok)
    torch.cuda.synchronize()
    if record:
        band_rows = {k: np.stack(v) for k, v in band_rows.items()}
        kv_rows = {b: (np.stack(K), np.stack(V)) for b, (K, V) in kv_rows.items()}
    return DecodeResult(torch.stack(out_tokens, 1).cpu().numpy(), n_cache.cpu().tolist(), evictions, band_rows,
                        kv_rows, ctx, cache)


def main():
    p = argparse.ArgumentParser()
    p.add_argument("--layers", type=int, default=32)
    p.add_argument("--hidden", type=int, default=4096)
    p.add_argument("--batch", type=int, default=4)
    p.add_argument("--steps", type=int, default=256)
    p.add_argument("--budget", type=int, default=128)
    p.add_argument("--small", action="store_true", help="an 8-layer, 512-wide model")
    a = p.parse_args()
    shape = small_shape() if a.small else ModelShape(layers=a.layers, hidden=a.hidden)
    import time
    t0 = time.time()
    r = decode(shape, batch=a.batch, steps=a.steps, budget=a.budget)
    dt = time.time() - t0
    st, code = E.epikv_get_error(r.ctx)
    print(f"decoded {a.batch} x {a.steps} tokens in {dt:.1f} s; cache lengths {r.n_cache}; "
          f"{r.evictions} evictions; device error {code}")


if __name__ == "__main__":
    main()
