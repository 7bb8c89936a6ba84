"""The five synthetic decode workloads and the small test shapes.

Each workload fixes the model shape, the trace lengths, the budget K, the
eviction schedule and the KV layout.  Sizes mirror the paper's setting
(a 32-layer model with 8 KV heads of dimension 128 and hidden size 4096,
reasoning traces of ~4k-32k tokens, budgets 512-8192, Sec. 3.5); the data
are seeded and synthetic (``synth.gen``): no benchmark item is used.
"""
from __future__ import annotations

import dataclasses

from .gen import TraceModel, seq_choice, seq_length

BANDZ = 1
LAGKV = 2
CONTIGUOUS = 0
PAGED = 1


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    model: TraceModel
    n_seq: int
    lengths: tuple          # trace length per sequence
    budgets: tuple          # K per sequence
    policies: tuple         # score kind that drives selection, per sequence
    kinds: int              # score kinds computed by every update
    chunk: int              # new tokens per sequence per update call
    trigger_slack: tuple    # evict when n_cache > K + slack
    layout: int
    block_size: int = 16
    z_window: int = 64
    lag: int = 16
    lag_window: int = 64
    recency_cap: int = 128
    prefill: tuple = ()     # prefill length per sequence (0 = pure decode)

    @property
    def max_len(self):
        return max(self.lengths)

    def prefill_len(self, b):
        return self.prefill[b] if self.prefill else 0


def config(i: int) -> Workload:
    """Workload ``i`` (1..5) at full size."""
    seed = 0xE91C0000 + i
    if i == 1:
        # one sequence, 2,048 tokens scored in one call, one eviction to K=512
        return Workload("single_2k_bandz_K512", TraceModel(seed), 1, (2048,), (512,), (BANDZ,),
                        BANDZ, 2048, (0,), CONTIGUOUS)
    if i == 2:
        # batch 8 x 8,192 tokens, band score, evict every 64 tokens to K=4096
        return Workload("batch8_8k_bandz_K4096", TraceModel(seed), 8, (8192,) * 8, (4096,) * 8,
                        (BANDZ,) * 8, BANDZ, 64, (63,) * 8, CONTIGUOUS)
    if i == 3:
        # batch 32 x 32,768 tokens, Lag-KV (lag 16), paged 16-token blocks, evict every 128 to K=8192
        return Workload("batch32_32k_lagkv_paged_K8192", TraceModel(seed), 32, (32768,) * 32,
                        (8192,) * 32, (LAGKV,) * 32, LAGKV, 128, (127,) * 32, PAGED)
    if i == 4:
        # batch 4 x 65,536 tokens, per-token score updates, one eviction to K=4096
        return Workload("batch4_64k_bandz_K4096", TraceModel(seed), 4, (65536,) * 4, (4096,) * 4,
                        (BANDZ,) * 4, BANDZ, 1, (65536,) * 4, CONTIGUOUS)
    if i == 5:
        # ragged continuous decode: 64 sequences of 4k-32k tokens, budgets from {2048, 4096, 8192},
        # evict a sequence when its cache exceeds K + 64; both scores every step
        n = 64
        lengths = tuple(seq_length(seed, b, 4096, 32768) for b in range(n))
        budgets = tuple(seq_choice(seed, b, (2048, 4096, 8192)) for b in range(n))
        policies = tuple(BANDZ if b % 2 == 0 else LAGKV for b in range(n))
        return Workload("ragged64_4k32k_both_paged", TraceModel(seed), n, lengths, budgets, policies,
                        BANDZ | LAGKV, 1, (64,) * n, PAGED)
    raise ValueError(i)


def small_model(seed: int) -> TraceModel:
    """A reduced model for parity tests that the oracle finishes in seconds."""
    return TraceModel(seed, num_layers=4, hidden=256, num_kv_heads=2, head_dim=32,
                      band_a=(1,), band_b=(2, 3))


def pyramid_budgets(k_mean: int, n_layers: int, spread: float = 0.5, multiple: int = 16) -> tuple:
    """A per-layer budget vector for the per-layer budget workloads: larger
    budgets for lower layers, falling linearly from (1 + spread) * k_mean at
    layer 0 to (1 - spread) * k_mean at the last layer, each rounded to a
    multiple of ``multiple`` (so the mean stays k_mean)."""
    out = []
    for l in range(n_layers):
        f = 1.0 + spread * (1.0 - 2.0 * l / (n_layers - 1)) if n_layers > 1 else 1.0
        out.append(int(round(k_mean * f / multiple)) * multiple)
    return tuple(out)
