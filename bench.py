#!/usr/bin/env python
"""Throughput of the EpiKV eviction hot path on GB300.

Headline workload (the 32k-context decode configuration): 32 sequences per
GPU, 32 layers x 8 KV heads x 128 dims bf16 K/V in a paged pool of 16-token
blocks with shuffled block tables, budget K = 8192, Lag-KV scores (lag 16,
rolling window 64).  One step = the steady-state decode chunk of every
sequence: 128 new tokens per sequence are scored, each cache (8,320 tokens)
is cut back to K and every layer's K and V are compacted in place -- one
epikv_step through the C ABI (Lag-KV partial kernel, finalize kernel, select
kernel, TMA compaction kernel).

Inputs are resident in HBM before timing: the 8,192-token caches and the new
tokens of every timed step (pre-generated into fresh pool blocks that each
step's block table points to, as a paged serving loop appends tokens).  The
cache and pool (tens of GB) are far larger than L2, so no flush is needed.

`value` = tokens scored per second over the timed steps (all ranks);
`e2e` = the same steps again through the same call, from the same state (the
workspace and resident caches are restored), with each step's new K/V copied
from pinned host memory and the new cache lengths read back;
`roofline` = the compaction kernel's algorithmic bytes (2 x moved rows x
128 KiB) per launch over its CUDA-event duration, against the measured HBM
copy bandwidth; `configs` = the five workloads measured one after another
(single GPU), each with its kernels' CUDA-event times and HBM fractions.
Under torchrun every rank owns its own sequences (global ids rank * 32 ..
rank * 32 + 31): the batch is sharded by sequence with no data exchange.
`--impl reference` times the fp64 CPU oracle instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "eviction tokens/s (score+z+top-K+compact)"
UNIT = "tokens/s"
WORKLOAD = "batch32_32k_lagkv_paged16_K8192_chunk128"


def parse(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    # skip the per-configuration table of the default run
    p.add_argument("--no-configs", action="store_true")
    # CTAs of the end-to-end measurement's host-to-device upload kernel
    p.add_argument("--upload-ctas", type=int, default=32)
    # a scaled-down variant of the same workload, for profiler captures
    p.add_argument("--sequences", type=int, default=32)
    p.add_argument("--budget", type=int, default=8192)
    p.add_argument("--chunk", type=int, default=128)
    # one workload alone (the per-configuration table runs them all):
    # bandz2k = configuration 1, bandz8k = 2, lagkv32k = 3 (default),
    # pertoken / evict64k = the two phases of 4, ragged64 = 5; layers32k =
    # per-layer budgets on configuration 3's shape
    p.add_argument("--workload", default="lagkv32k",
                   choices=["lagkv32k", "bandz2k", "pertoken", "evict64k", "layers32k", "bandz8k", "ragged64"])
    # K/V score kinds computed at the 32k workload (selection uses Lag-KV):
    # 2 = Lag-KV only; 58 = Lag-KV + KV-key + KV-val + lag-kv-key
    p.add_argument("--kinds", type=int, default=2)
    # chunk-level selection at the 32k workload: position chunks of this many
    # tokens (1 = the paper's token-level selection)
    p.add_argument("--select-chunk", type=int, default=1)
    # oracle processes of the CPU baseline (0: one per available core)
    p.add_argument("--cpu-workers", type=int, default=0)
    # a scaled-down variant of the decode-window workloads (bandz8k, ragged64)
    # for profiler captures: their first N sequences, and one budget for all
    p.add_argument("--window-seqs", type=int, default=0)
    p.add_argument("--window-budget", type=int, default=0)
    return p.parse_args(argv)


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), int(os.environ.get("WORLD_SIZE", 1))


def shard_sequences(per_rank, rank, world):
    """Global sequence ids owned by `rank` when a batch of per_rank * world
    sequences is split by sequence over `world` ranks: a contiguous block of
    per_rank ids.  Every sequence (its K/V, its workspace slots, its seeds)
    lives on exactly one rank, so ranks exchange no data."""
    assert 0 <= rank < world and per_rank >= 1
    return list(range(rank * per_rank, (rank + 1) * per_rank))


def aggregate_ranks(local_ms, units_per_rank, world, device=None):
    """Whole-job timing of sequence-sharded ranks: the slowest rank's duration
    and the units all ranks processed per second over it."""
    units = float(units_per_rank)
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([local_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        local_ms = float(t.item())
        u = torch.tensor([units], dtype=torch.float64, device=device)
        dist.all_reduce(u, op=dist.ReduceOp.SUM)
        units = float(u.item())
    return local_ms, units / (local_ms / 1e3)


def measured_hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def ncu_traffic(kernel):
    """ncu DRAM traffic of a launch as a ratio to its algorithmic bytes, from
    the committed summary, or None when the kernel's source changed since the
    counters were taken."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    src = os.path.join(ROOT, "paper_2606_26472_gb300", "csrc")
    h = hashlib.sha256()
    for f in ("compact.cu", "common.cuh"):
        h.update(open(os.path.join(src, f), "rb").read())
    for line in open(path):
        parts = line.split()
        if len(parts) == 3 and parts[0] == kernel and parts[1] == h.hexdigest()[:16]:
            return float(parts[2])
    return None


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during timing."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id   # the device's UUID ("GPU-...") so no other GPU is sampled
        self.proc = None

    @staticmethod
    def device_id(dev, local_rank):
        """nvidia-smi's --id for torch device `dev`: its UUID, else the local rank."""
        import torch
        try:
            uuid = str(torch.cuda.get_device_properties(dev).uuid)
            return uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            return str(local_rank)

    def start(self):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu_id}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.count(",") >= 8]
        os.unlink(self.f.name)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if "Active" == r[5 + i].strip()})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- CPU oracle
def oracle_sequence_step(seq, pos0):
    """One sequence's decode step of the 32k workload, timed on the fp64
    oracle: Lag-KV scores of 128 new tokens, full-sort selection over the
    8,320-slot cache and the gather of the kept K/V rows of every layer.  The
    rows are regenerated first, untimed.  Returns (tokens, seconds)."""
    from oracle import epikv_oracle as O
    from synth import gen, host, workloads as W

    wl = W.config(3)
    m = wl.model
    tabs = gen.make_tables(m)
    K, C, lag, w = wl.budgets[0], wl.chunk, wl.lag, wl.lag_window
    shape = (K + C, m.num_layers, m.num_kv_heads, m.head_dim)
    cache_k = np.ones(shape, np.uint16)       # gather cost does not depend on the bytes
    cache_v = np.ones(shape, np.uint16)
    first = (pos0 - (w - 1)) // lag * lag - lag  # rows the u window and its ranges reach
    positions = np.arange(first, pos0 + C)
    sp = gen.spike_flags(m, seq, pos0 + C)
    Kr = gen.bf16_bits_to_f64(host.kv_rows(m, tabs, seq, 0, positions, sp))
    Vr = gen.bf16_bits_to_f64(host.kv_rows(m, tabs, seq, 1, positions, sp))
    old = np.random.default_rng(seq).normal(size=K)   # frozen scores of the cached tokens
    t0 = time.perf_counter()
    u = {}
    for t in range(pos0 - (w - 1), pos0 + C):
        c = t // lag
        lo = (c - 1) * lag - first
        u[t] = O.lag_token_variance(Kr[t - first], Vr[t - first], Kr[lo:lo + lag], Vr[lo:lo + lag])
    s_new = [np.mean([u[t - k] for k in range(w)]) for t in range(pos0, pos0 + C)]
    scores = np.concatenate([old, s_new])
    kept = O.select_kept(scores, K, 0, wl.recency_cap)
    O.compact(cache_k, kept)
    O.compact(cache_v, kept)
    return C, time.perf_counter() - t0


def _oracle_task(job):
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    seq, pos0 = job
    tok, sec = oracle_sequence_step(seq, pos0)
    return os.getpid(), tok, sec


def oracle_workers(requested=0):
    n = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    return max(1, min(n, requested) if requested else n)


def oracle_pool(workers):
    """A pool of oracle processes (spawn: safe after CUDA use in this process)."""
    import multiprocessing as mp
    return mp.get_context("spawn").Pool(workers, initializer=_pool_init)


def oracle_batch(pool, jobs):
    """Oracle sequence-steps on the pool's processes.  Returns (tokens,
    seconds): the tokens of every job over the busiest process's summed
    compute time (the processes run concurrently)."""
    res = pool.map(_oracle_task, jobs, chunksize=1)
    busy = {}
    for pid, _, sec in res:
        busy[pid] = busy.get(pid, 0.0) + sec
    return sum(t for _, t, _ in res), max(busy.values())


def _pool_init():
    # one core per process: numpy's own threads would oversubscribe the host
    os.environ["OMP_NUM_THREADS"] = "1"
    os.environ["OPENBLAS_NUM_THREADS"] = "1"
    sys.path.insert(0, ROOT)


def cpu_baseline(requested_workers=0):
    """The fp64 oracle on the host's cores: the decode step of all 32 sequences
    of the 32k workload (one process per core, one sequence-step per task)."""
    workers = oracle_workers(requested_workers)
    with oracle_pool(workers) as pool:
        oracle_batch(pool, [(b, 8192) for b in range(workers)])          # warm-up: imports, first allocations
        tok, sec = oracle_batch(pool, [(b, 8192 + 128) for b in range(32)])
    return {"value": tok / sec, "unit": UNIT, "cores": workers, "kind": "oracle",
            "sample": f"32 of 32 sequences x 1 decode step (128 tokens each: fp64 Lag-KV u over 191 positions + "
                      f"rolling mean, full-sort selection over 8320 slots, gather of the 8192 kept K and V rows "
                      f"of 32 layers), numpy, one process per core on {workers} cores, rows generated untimed; "
                      f"time = the busiest process's compute, {sec:.1f} s"}


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return None
    workers = oracle_workers(args.cpu_workers)
    budget_s = 150.0
    tot_tok, tot_s, steps, warm = 0, 0.0, 0, 0
    with oracle_pool(workers) as pool:
        t0 = time.perf_counter()
        for _ in range(max(1, args.warmup)):   # untimed decode steps of the 32 sequences
            oracle_batch(pool, [(b, 8192 + 128) for b in range(32)])
            warm += 1
            if time.perf_counter() - t0 > budget_s / 3:
                break
        t0 = time.perf_counter()
        for i in range(max(1, args.steps)):
            t, s = oracle_batch(pool, [(b, 8192 + 128 * (i + 1)) for b in range(32)])
            tot_tok += t
            tot_s += s
            steps += 1
            if time.perf_counter() - t0 > budget_s:
                break
    v = tot_tok / tot_s
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
            "steps": steps, "warmup": warm, "ms_per_step": 1e3 * tot_s / steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "oracle_step": "the decode step of all 32 sequences"},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": workers, "kind": "oracle",
                             "sample": f"{steps} decode steps of the 32 sequences, numpy fp64, one process per "
                                       f"core on {workers} cores"},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return line


# --------------------------------------------------------------------------- GPU helpers
def gpu_device(local_rank=0):
    import torch

    from paper_2606_26472_gb300 import build as B
    from paper_2606_26472_gb300 import epikv as E
    torch.cuda.set_device(local_rank)
    if not os.path.exists(E.LIB_PATH):
        B.build()
    E.load()
    return torch.device("cuda", local_rank)


def stream_bytes(m, *, tokens, seq_calls, rows_moved, kinds, one_token):
    """Algorithmic HBM bytes of the streaming kernels over a pass that scored
    `tokens` tokens in `seq_calls` (sequence, call) pairs and moved
    `rows_moved` token rows (all layers' K and V):
    * a token's band rows (15 x 4096 bf16) are read once; a chunked call also
      reads and writes each sequence's saved previous rows (h_prev), a
      one-token call reads its new rows and h_prev and writes h_prev;
    * a token's K and V rows of every layer are read once; with a Lag-KV kind
      each (sequence, call) also reads and writes its range state
      ([L][K|V][4][H][d] bf16);
    * the compaction reads and writes every moved row."""
    nb, D = len(m.band_layers), m.hidden
    L, H, d = m.num_layers, m.num_kv_heads, m.head_dim
    band_row = nb * D * 2
    kv_row = L * 2 * H * d * 2
    rng_state = L * 2 * 4 * H * d * 2
    band = bool(kinds & (1 | 4))
    kv = bool(kinds & (2 | 8 | 16 | 32))
    state = 2 * rng_state if kinds & (2 | 32) else 0
    out = {"compact_kernel": 2 * rows_moved * kv_row}
    if one_token:
        if kv:
            out["token_kernel"] = seq_calls * ((3 * band_row if band else 0) + kv_row + state)
        elif band:
            out["bandz_token_kernel"] = seq_calls * 3 * band_row
    else:
        if band:
            out["bandz_g_kernel"] = tokens * band_row + seq_calls * 2 * band_row
        if kv:
            out["lagkv_partial_kernel"] = tokens * kv_row + seq_calls * state
    return out


def kernel_table(records, n_steps, bytes_per_pass, peak):
    """Per-kernel CUDA-event times of a pass of n_steps steps (records: [(name,
    ms)] from epikv_set_kernel_events) -> {kernel: launches and ms per step,
    and for the HBM-streaming kernels their algorithmic GB/s and fraction of
    the measured copy bandwidth}."""
    from paper_2606_26472_gb300 import epikv as E
    acc = {}
    for name, ms in records:
        a = acc.setdefault(E.kernel_short_name(name), [0, 0.0])
        a[0] += 1
        a[1] += ms
    tab = {}
    for k, (n, ms) in acc.items():
        e = {"launches_per_step": n / n_steps, "ms_per_step": ms / n_steps}
        b = bytes_per_pass.get(k)
        if b and ms > 0:
            gbs = b / (ms / 1e3) / 1e9
            e.update(algorithmic_bytes_per_step=b / n_steps, gbs=gbs, hbm_frac=gbs / peak)
        tab[k] = e
    return tab


def kernel_pass(E, ctx, n_launches, run):
    """Run `run()` with every kernel of `ctx` bracketed by events; [(name, ms)]."""
    kc = E.KernelClock(ctx, n_launches)
    kc.start()
    try:
        run()
    finally:
        recs = kc.stop()
    return recs


# --------------------------------------------------------------------------- configuration 3 (headline)
def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2606_26472_gb300 import epikv as E
    from paper_2606_26472_gb300.cache import KVCache
    from synth import gen, workloads as W
    from synth.device import DeviceTrace, upload_2d

    rank, local_rank, world = dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    dev = gpu_device(local_rank)

    wl = W.config(3)
    m = wl.model
    Bn, K, C = args.sequences, args.budget, args.chunk
    assert K % wl.block_size == 0 and C % wl.block_size == 0
    gids = shard_sequences(Bn, rank, world)     # this rank's global sequence ids (generator seeds)
    workload = WORKLOAD if (Bn, K, C) == (wl.n_seq, wl.budgets[0], wl.chunk) else \
        f"batch{Bn}_lagkv_paged16_K{K}_chunk{C}"
    if args.kinds != E.EPIKV_SCORE_LAGKV:
        workload += f"_kinds{args.kinds}"
    if args.select_chunk > 1:
        workload += f"_selectchunk{args.select_chunk}"
    L, H, d = m.num_layers, m.num_kv_heads, m.head_dim
    bs = wl.block_size
    T_cap = K + C
    mb = T_cap // bs
    common = K // bs
    fresh = C // bs
    kc_steps = 3                                  # the per-kernel pass after the timed steps
    n_steps = args.warmup + args.steps + kc_steps
    e2e_on = not args.no_e2e
    n_blocks = Bn * common + n_steps * Bn * fresh + (2 * Bn * fresh if e2e_on else 0)
    perm = gen.block_permutation(m.seed ^ rank, Bn * common).reshape(Bn, common)

    def table(fresh_base):
        bt = np.empty((Bn, mb), np.int32)
        bt[:, :common] = perm
        bt[:, common:] = fresh_base + np.arange(Bn * fresh, dtype=np.int32).reshape(Bn, fresh)
        return torch.from_numpy(bt).to(dev)

    tables = [table(Bn * common + st * Bn * fresh) for st in range(n_steps)]
    e2e_base = Bn * common + n_steps * Bn * fresh
    cache = KVCache(E.EPIKV_LAYOUT_PAGED, L, H, d, max_seqs=Bn, max_tokens=T_cap, block_size=bs,
                    num_blocks=n_blocks, block_table=tables[0].cpu().numpy(), device=dev)
    dt = DeviceTrace(m, dev)
    stream = torch.cuda.current_stream()

    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=T_cap, max_new_tokens=C, num_layers=L, num_kv_heads=H,
                        head_dim=d, lag=wl.lag, lag_window=wl.lag_window, recency_cap=wl.recency_cap,
                        score_kinds=args.kinds, select_chunk=args.select_chunk)
    assert args.kinds & E.EPIKV_SCORE_LAGKV and not args.kinds & (E.EPIKV_SCORE_BANDZ | E.EPIKV_SCORE_HSVAR)
    ws_bytes = E.epikv_workspace_bytes(cfg)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    ctx = E.epikv_init(cfg, ws, ws_bytes)
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_LAGKV)

    # the first K tokens of every trace, scored in decode chunks (no eviction yet)
    for b in range(Bn):
        dt.kv(gids[b], 0, K, 0, cache.k, cache.v, **cache.synth_kwargs(tables[0]))
    seq_ids = torch.arange(Bn, dtype=torch.int32, device=dev)
    cu_new = (torch.arange(Bn + 1, dtype=torch.int32, device=dev) * C).contiguous()
    view0 = cache.view(tables[0])
    for _ in range(K // C):
        E.epikv_score_update(ctx, Bn, seq_ids, cu_new, C, None, view0)
    # every step's new tokens, appended into fresh blocks before timing
    for st in range(n_steps):
        for b in range(Bn):
            dt.kv(gids[b], K + st * C, C, K, cache.k, cache.v, **cache.synth_kwargs(tables[st]))
    views = [cache.view(t) for t in tables]
    budget = torch.full((Bn,), K, dtype=torch.int32, device=dev)
    trigger = torch.full((Bn,), K + C - 1, dtype=torch.int32, device=dev)
    n_out = torch.empty(Bn, dtype=torch.int32, device=dev)
    torch.cuda.synchronize()
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code} during set-up"

    def step(view):
        E.epikv_step(ctx, Bn, seq_ids, cu_new, C, budget, trigger, None, view, n_out)

    for st in range(args.warmup):
        step(views[st])
    torch.cuda.synchronize()
    # the state before the timed steps, restored for the end-to-end pass so that
    # it repeats the same steps (same kept lists, same rows moved)
    snap = None
    if e2e_on:
        snap = (ws.clone(), cache.k[:, :Bn * common].clone(), cache.v[:, :Bn * common].clone())
    stats0 = E.epikv_get_stats(ctx)

    def new_events():
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        for e in evs:
            e.record(stream)   # materialise the handles
        return evs

    phase = [new_events() for _ in range(args.steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    clocks = Clocks(Clocks.device_id(dev, local_rank)).start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    for i in range(args.steps):
        E.epikv_set_phase_events(ctx, phase[i])
        step(views[args.warmup + i])
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    E.epikv_set_phase_events(ctx, None)
    ms = t_start.elapsed_time(t_end)
    stats1 = E.epikv_get_stats(ctx)
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code}"
    t_score = sum(p[0].elapsed_time(p[1]) for p in phase)
    t_select = sum(p[1].elapsed_time(p[2]) for p in phase)
    per_compact = sorted(p[2].elapsed_time(p[3]) for p in phase)
    t_compact = sum(per_compact)
    rows_moved = stats1["rows_moved"] - stats0["rows_moved"]
    tokens = stats1["tokens_scored"] - stats0["tokens_scored"]
    assert tokens == Bn * C * args.steps
    row_bytes = L * 2 * H * d * 2                       # one token's K and V, all layers
    compact_bytes = 2 * rows_moved * row_bytes           # read + write
    score_bytes = sum(stream_bytes(m, tokens=tokens, seq_calls=Bn * args.steps, rows_moved=0, kinds=args.kinds,
                                   one_token=False).values())
    peak, peak_src = measured_hbm_peak()

    # per-kernel CUDA-event times: the next kc_steps steps, every kernel bracketed by events
    s_k0 = E.epikv_get_stats(ctx)
    recs = kernel_pass(E, ctx, 8 * kc_steps, lambda: [step(views[args.warmup + args.steps + j])
                                                      for j in range(kc_steps)])
    s_k1 = E.epikv_get_stats(ctx)
    kernels = kernel_table(recs, kc_steps,
                           stream_bytes(m, tokens=Bn * C * kc_steps, seq_calls=Bn * kc_steps,
                                        rows_moved=s_k1["rows_moved"] - s_k0["rows_moved"], kinds=args.kinds,
                                        one_token=False), peak)

    ms, value = aggregate_ranks(ms, tokens, world, dev)

    # ---- end to end: the timed steps again, from the same state, with each
    # step's new K/V copied from pinned host memory and its new lengths read back
    e2e = None
    if e2e_on:
        ws.copy_(snap[0])
        cache.k[:, :Bn * common].copy_(snap[1])
        cache.v[:, :Bn * common].copy_(snap[2])
        del snap
        # two sets of fresh blocks: step i+1's K/V are copied in on a side
        # stream while step i runs, as a serving loop would overlap them
        tabs = [table(e2e_base + j * Bn * fresh) for j in range(2)]
        views_e = [cache.view(t) for t in tabs]
        n_e = args.steps
        payload = [torch.empty((2, L, Bn * fresh, bs, H, d), dtype=torch.bfloat16, pin_memory=True)
                   for _ in range(n_e)]
        lo = e2e_base
        for j in range(n_e):     # timed step j's new tokens, generated again, kept on the host
            for b in range(Bn):
                dt.kv(gids[b], K + (args.warmup + j) * C, C, K, cache.k, cache.v, **cache.synth_kwargs(tabs[0]))
            payload[j][0].copy_(cache.k[:, lo:lo + Bn * fresh])
            payload[j][1].copy_(cache.v[:, lo:lo + Bn * fresh])
        lens = torch.empty((n_e, (Bn + 3) // 4 * 4), dtype=torch.int32, pin_memory=True)   # 16-byte rows
        copy_stream = torch.cuda.Stream(device=dev)
        copied = [torch.cuda.Event(enable_timing=True) for _ in range(n_e)]
        stepped = [torch.cuda.Event(enable_timing=True) for _ in range(n_e)]
        copy_start = [torch.cuda.Event(enable_timing=True) for _ in range(n_e)]
        step_start = [torch.cuda.Event(enable_timing=True) for _ in range(n_e)]

        # one strided upload per K and V and step (32 layer planes of 8 MiB
        # each), read from the pinned host buffer by SM loads over the host
        # link: the copy engines of this platform stall every ~0.5 s for
        # ~0.1 s, the SM path does not (both move ~210 GB/s otherwise)
        plane = Bn * fresh * bs * H * d * 2                 # bytes of one layer's new rows
        pitch = cache.k.stride(0) * 2                       # bytes between layer planes of the pool
        up_ctas = args.upload_ctas

        def h2d(i):   # step i's new K/V into block set i % 2, after step i-2 released it
            lo_i = e2e_base + (i % 2) * Bn * fresh
            if i >= 2:
                copy_stream.wait_event(stepped[i - 2])
            copy_start[i].record(copy_stream)
            src = payload[i]
            for kind, pool in ((0, cache.k), (1, cache.v)):
                upload_2d(pool[0, lo_i].data_ptr(), pitch, src[kind].data_ptr(), plane, plane, L, up_ctas, copy_stream)
            copied[i].record(copy_stream)

        # the copy kernel's first launch (module load, first transfers) before timing
        for kind, pool in ((0, cache.k), (1, cache.v)):
            upload_2d(pool[0, e2e_base + Bn * fresh].data_ptr(), pitch, payload[0][kind].data_ptr(), plane, plane, L,
                      up_ctas, copy_stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        stats_e0 = E.epikv_get_stats(ctx)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        copy_stream.wait_event(e0)
        h2d(0)
        for i in range(n_e):
            if i + 1 < n_e:
                h2d(i + 1)
            stream.wait_event(copied[i])
            step_start[i].record(stream)
            step(views_e[i % 2])
            stepped[i].record(stream)
            # the new lengths read back by SM stores into pinned host memory (the
            # copy engines' occasional stalls would hold the stream)
            upload_2d(lens[i].data_ptr(), lens.stride(0) * 4, n_out.data_ptr(), Bn * 4, Bn * 4, 1, 1, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        stats_e1 = E.epikv_get_stats(ctx)
        e_tokens = stats_e1["tokens_scored"] - stats_e0["tokens_scored"]
        e_ms, e_value = aggregate_ranks(e0.elapsed_time(e1), e_tokens, world, dev)
        assert (lens.numpy()[:, :Bn] == K).all()
        copy_ms = sorted(copy_start[i].elapsed_time(copied[i]) for i in range(n_e))
        step_ms = sorted(step_start[i].elapsed_time(stepped[i]) for i in range(n_e))
        rows_e = stats_e1["rows_moved"] - stats_e0["rows_moved"]
        e2e = {"value": e_value, "unit": UNIT,
               "h2d_bytes_per_step": int(payload[0].numel() * 2), "d2h_bytes_per_step": Bn * 4,
               "steps": n_e,
               "same_steps_as_timed": "the timed steps repeated from the restored pre-timing state",
               "overlap": "step i+1's host-to-device upload (SM loads of pinned host memory) runs on a side stream "
                          "during step i",
               "median_ms": {"h2d_copy": copy_ms[len(copy_ms) // 2], "step": step_ms[len(step_ms) // 2],
                             "wall_per_step": e_ms / n_e},
               "max_ms": {"h2d_copy": copy_ms[-1], "step": step_ms[-1]},
               "slow_copies": sum(c > 2 * copy_ms[len(copy_ms) // 2] for c in copy_ms),
               "rows_moved_per_step": rows_e / n_e,
               "rows_moved_match_timed": rows_e == rows_moved}
        st_, code = E.epikv_get_error(ctx)
        assert st_ == E.EPIKV_OK, f"device error {code} in e2e"
        del payload

    E.epikv_destroy(ctx)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return None
    ach = compact_bytes / args.steps / (t_compact / args.steps / 1e3) / 1e9
    ratio = ncu_traffic("compact_kernel")
    traffic = None if ratio is None else ratio * compact_bytes / args.steps
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": workload, "sequences": Bn, "global_batch": Bn * world, "context": 32768,
                   "budget_K": K, "chunk": C, "layers": L, "kv_heads": H, "head_dim": d, "kv_dtype": "bf16",
                   "layout": "paged16_shuffled", "score": "lagkv_lag16_w64", "select_chunk": args.select_chunk,
                   "parallelism": f"sequence-sharded x{world} (rank r owns global sequences {Bn}r..{Bn}r+{Bn - 1})",
                   "l2": "inputs larger than L2 (paged pool %.1f GiB)" % (cache.k.numel() * 4 / 2 ** 30)},
        "compaction_gbs": ach,
        "rows_moved_per_step": rows_moved / args.steps,
        "kernels_ms_per_step": {"score": t_score / args.steps, "select": t_select / args.steps,
                                "compact": t_compact / args.steps},
        "compact_ms_min_median_max": [per_compact[0], per_compact[len(per_compact) // 2], per_compact[-1]],
        "step_hbm_gbs": (compact_bytes + score_bytes) / (ms / 1e3) / 1e9 if world == 1 else None,
        "roofline": {"bound": "hbm", "kernel": "compact_kernel", "achieved": ach, "peak": peak, "unit": "GB/s",
                     "frac": ach / peak, "peak_source": peak_src,
                     "timed": "the compaction phase of every timed step (CUDA events on the launch stream around "
                              "compact_stash_kernel + compact_kernel + compact_consumed_kernel)",
                     "traffic": traffic, "algorithmic_bytes_per_launch": compact_bytes / args.steps},
        "kernels": kernels,
        "kernels_note": f"per-kernel CUDA events over {kc_steps} further steps, each kernel bracketed by events "
                        "(which also stops the early launch of the next kernel)",
        "gpu_launches": 6 * args.steps,   # Lag-KV partial, finalize, select, stash, compaction, eviction consumed
        "clocks": clk,
        "e2e": e2e,
    }
    if world > 1:
        dist.destroy_process_group()
    return line


# --------------------------------------------------------------------------- configuration 1
def run_bandz2k(args, steps=None, warmup=None):
    """Configuration 1.  One step = a fresh sequence: its 2,048 tokens scored
    with the band-z score (15 band layers of 4096 bf16), the cache cut to
    K = 512, all 32 layers' K/V compacted -- epikv_step on one sequence.
    Each step's sequence has its own resident cache and hidden rows."""
    import torch

    from paper_2606_26472_gb300 import epikv as E
    from paper_2606_26472_gb300.cache import KVCache
    from synth import workloads as W
    from synth.device import DeviceTrace

    _, local_rank, world = dist_env()
    assert world == 1, "the band-z workload is a single-GPU measurement"
    dev = gpu_device(local_rank)
    steps = args.steps if steps is None else steps
    warmup = args.warmup if warmup is None else warmup
    kc_steps = 3
    wl = W.config(1)
    m = wl.model
    T, K = wl.max_len, wl.budgets[0]
    S = warmup + steps + kc_steps
    nb = len(m.band_layers)
    dt = DeviceTrace(m, dev)
    cache = KVCache(E.EPIKV_LAYOUT_CONTIGUOUS, m.num_layers, m.num_kv_heads, m.head_dim, max_seqs=S, max_tokens=T,
                    device=dev)
    hid = torch.empty((nb, S, T, m.hidden), dtype=torch.bfloat16, device=dev)
    for s_ in range(S):
        dt.kv(s_, 0, T, 0, cache.k, cache.v, **cache.synth_kwargs())
        for i, layer in enumerate(m.band_layers):
            dt.hidden(s_, layer, 0, T, hid[i, s_], m.hidden)
    cfg = E.make_config(max_seqs=S, max_cache_tokens=T, max_new_tokens=T, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), score_kinds=E.EPIKV_SCORE_BANDZ)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device=dev)
    ctx = E.epikv_init(cfg, ws, ws.numel())
    kv = cache.view()
    views = [E.hidden_view([hid[i, s_] for i in range(nb)], m.hidden) for s_ in range(S)]
    ids = [torch.tensor([s_], dtype=torch.int32, device=dev) for s_ in range(S)]
    cu = torch.tensor([0, T], dtype=torch.int32, device=dev)
    budget = torch.tensor([K], dtype=torch.int32, device=dev)
    trigger = torch.tensor([K], dtype=torch.int32, device=dev)
    n_out = torch.empty(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    for s_ in range(S):
        E.epikv_seq_reset(ctx, s_, 0, E.EPIKV_SCORE_BANDZ)

    def step(s_):
        E.epikv_step(ctx, 1, ids[s_], cu, T, budget, trigger, views[s_], kv, n_out)

    for s_ in range(warmup):
        step(s_)
    torch.cuda.synchronize()
    stats0 = E.epikv_get_stats(ctx)
    phase = []
    for _ in range(steps):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        for e in evs:
            e.record(stream)
        phase.append(evs)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clocks = Clocks(Clocks.device_id(dev, local_rank)).start()
    torch.cuda.synchronize()
    t0.record(stream)
    for i in range(steps):
        E.epikv_set_phase_events(ctx, phase[i])
        step(warmup + i)
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    E.epikv_set_phase_events(ctx, None)
    ms = t0.elapsed_time(t1)
    stats1 = E.epikv_get_stats(ctx)
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code}"
    tokens = stats1["tokens_scored"] - stats0["tokens_scored"]
    rows = stats1["rows_moved"] - stats0["rows_moved"]
    t_score = sum(p[0].elapsed_time(p[1]) for p in phase) / steps
    t_select = sum(p[1].elapsed_time(p[2]) for p in phase) / steps
    t_compact = sum(p[2].elapsed_time(p[3]) for p in phase) / steps
    sb = stream_bytes(m, tokens=T, seq_calls=1, rows_moved=rows / steps, kinds=E.EPIKV_SCORE_BANDZ, one_token=False)
    score_bytes, compact_bytes = sb["bandz_g_kernel"], sb["compact_kernel"]
    peak, peak_src = measured_hbm_peak()
    g = score_bytes / (t_score / 1e3) / 1e9
    c = compact_bytes / (t_compact / 1e3) / 1e9
    s_k0 = E.epikv_get_stats(ctx)
    recs = kernel_pass(E, ctx, 8 * kc_steps, lambda: [step(warmup + steps + j) for j in range(kc_steps)])
    s_k1 = E.epikv_get_stats(ctx)
    kernels = kernel_table(recs, kc_steps, stream_bytes(m, tokens=T * kc_steps, seq_calls=kc_steps,
                                                        rows_moved=s_k1["rows_moved"] - s_k0["rows_moved"],
                                                        kinds=E.EPIKV_SCORE_BANDZ, one_token=False), peak)
    E.epikv_destroy(ctx)
    return {"metric": METRIC, "value": tokens / (ms / 1e3), "unit": UNIT, "n_gpus": 1, "steps": steps,
            "warmup": warmup, "ms_per_step": ms / steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": "single_2k_bandz_K512_fresh_sequence_per_step", "band_layers": nb,
                       "hidden": m.hidden, "budget_K": K, "layout": "contiguous",
                       "step": "one fresh sequence: 2,048 tokens scored, one eviction 2,048 -> 512",
                       "l2": "inputs larger than L2 (%.1f GiB resident)" % ((cache.k.numel() * 2 + hid.numel()) * 2 / 2 ** 30)},
            "kernels_ms_per_step": {"score": t_score, "select": t_select, "compact": t_compact},
            "score_phase_gbs": g, "compaction_gbs": c, "compaction_frac": c / peak,
            "roofline": {"bound": "hbm", "kernel": "score phase (bandz_g_kernel + score_finalize_kernel)",
                         "achieved": g, "peak": peak, "unit": "GB/s", "frac": g / peak, "peak_source": peak_src,
                         "traffic": None, "algorithmic_bytes_per_launch": score_bytes},
            "kernels": kernels,
            "gpu_launches": 6 * steps,   # g, finalize, select, stash, compaction, eviction consumed
            "clocks": clk}


# --------------------------------------------------------------------------- configuration 4
def run_pertoken(args, steps=None, warmup=None):
    """Configuration 4's per-token phase: 4 sequences, one new token each per
    decode step, 15 band rows per token.  One bench step = 64 decode steps,
    issued either call by call or as one CUDA graph of 64
    epikv_score_update calls (the per-step kernels are tiny, so launch
    overhead decides the rate)."""
    import torch

    from paper_2606_26472_gb300 import epikv as E
    from synth import workloads as W
    from synth.device import DeviceTrace

    _, local_rank, world = dist_env()
    assert world == 1, "the per-token workload is a single-GPU measurement"
    dev = gpu_device(local_rank)
    steps = args.steps if steps is None else steps
    warmup = args.warmup if warmup is None else warmup
    wl = W.config(4)
    m = wl.model
    Bn, G = wl.n_seq, 64
    n_tok = (2 * (warmup + steps) + 2) * G     # eager run, graph run, the per-kernel block
    nb = len(m.band_layers)
    dt = DeviceTrace(m, dev)
    hid = torch.empty((nb, n_tok, Bn, m.hidden), dtype=torch.bfloat16, device=dev)
    for i, layer in enumerate(m.band_layers):
        for b in range(Bn):
            dt.hidden(b, layer, 0, n_tok, hid[i, :, b].data_ptr(), Bn * m.hidden)
    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=n_tok, max_new_tokens=1, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), score_kinds=E.EPIKV_SCORE_BANDZ)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device=dev)
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_BANDZ)
    seq_ids = torch.arange(Bn, dtype=torch.int32, device=dev)
    cu = torch.arange(Bn + 1, dtype=torch.int32, device=dev)
    step_bytes = Bn * m.hidden * 2
    bases = [hid[i].data_ptr() for i in range(nb)]
    kv_unused = E.kv_view(hid, hid, stride_layer=0, stride_seq=0, stride_token=1024)

    def view(t):
        hv = E.epikv_hidden_view()
        hv.row_stride = m.hidden
        for i in range(nb):
            hv.band_rows[i] = bases[i] + t * step_bytes
        return hv

    views = [view(t) for t in range(n_tok)]
    stream = torch.cuda.current_stream()
    t = 0
    E.epikv_score_update(ctx, Bn, seq_ids, cu, 1, views[t], kv_unused)
    t += 1

    def eager_block(t0):
        for k in range(G):
            E.epikv_score_update(ctx, Bn, seq_ids, cu, 1, views[t0 + k], kv_unused)

    def timed(run_block, t0):
        for w in range(warmup):
            run_block(t0 + w * G)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(steps):
            run_block(t0 + (warmup + i) * G)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    ms_eager = timed(eager_block, t)
    t += (warmup + steps) * G
    graphs = {}
    for blk in range(warmup + steps):     # one graph per 64-token block, captured before timing
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            eager_block(t + blk * G)
        graphs[t + blk * G] = g
    clocks = Clocks(Clocks.device_id(dev, local_rank)).start()
    ms_graph = timed(lambda t0: graphs[t0].replay(), t)
    clk = clocks.stop()
    t += (warmup + steps) * G
    peak, _ = measured_hbm_peak()
    recs = kernel_pass(E, ctx, G, lambda: eager_block(t))
    kernels = kernel_table(recs, 1, stream_bytes(m, tokens=G * Bn, seq_calls=G * Bn, rows_moved=0,
                                                 kinds=E.EPIKV_SCORE_BANDZ, one_token=True), peak)
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code}"
    E.epikv_destroy(ctx)
    tokens = steps * G * Bn
    return {"metric": METRIC, "value": tokens / (ms_graph / 1e3), "unit": UNIT, "n_gpus": 1, "steps": steps,
            "warmup": warmup, "ms_per_step": ms_graph / steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": "batch4_bandz_per_token_updates", "sequences": Bn, "band_layers": nb,
                       "hidden": m.hidden, "step": "64 decode tokens per sequence (one CUDA graph of 64 calls)",
                       "l2": "band rows of every token resident, %.1f GiB" % (hid.numel() * 2 / 2 ** 30)},
            "per_token_us": {"graph": 1e3 * ms_graph / (steps * G), "eager": 1e3 * ms_eager / (steps * G)},
            "eager_value": tokens / (ms_eager / 1e3),
            "kernels": kernels,
            "gpu_launches": G * steps,   # one fused g + z launch per decode step
            "clocks": clk}


def run_evict64k(args, steps=None, warmup=None):
    """Configuration 4's eviction phase: 4 sequences of 65,536 scored tokens
    (band-z), each cut to K = 4,096 at once -- the radix select over 65,408
    candidates per sequence (keys not staged in shared memory) and the
    compaction of every layer's K and V.  Each timed eviction starts from the
    same state: the workspace and the caches are restored (untimed) from a
    device snapshot taken after scoring."""
    import torch

    from paper_2606_26472_gb300 import epikv as E
    from paper_2606_26472_gb300.cache import KVCache
    from synth import workloads as W
    from synth.device import DeviceTrace

    _, local_rank, world = dist_env()
    assert world == 1, "the eviction workload is a single-GPU measurement"
    dev = gpu_device(local_rank)
    steps = min(args.steps, 5) if steps is None else steps
    warmup = min(args.warmup, 2) if warmup is None else warmup
    wl = W.config(4)
    m = wl.model
    Bn, T, K = wl.n_seq, wl.max_len, wl.budgets[0]
    L, H, d, nb = m.num_layers, m.num_kv_heads, m.head_dim, len(m.band_layers)
    CH = 4096                                       # tokens per scoring call (chunking does not change scores)
    dt = DeviceTrace(m, dev)
    cache = KVCache(E.EPIKV_LAYOUT_CONTIGUOUS, L, H, d, max_seqs=Bn, max_tokens=T, device=dev)
    for b in range(Bn):
        dt.kv(b, 0, T, 0, cache.k, cache.v, **cache.synth_kwargs())
    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=T, max_new_tokens=CH, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), score_kinds=E.EPIKV_SCORE_BANDZ)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device=dev)
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_BANDZ)
    kv = cache.view()
    hid = torch.empty((nb, Bn * CH, m.hidden), dtype=torch.bfloat16, device=dev)
    hv = E.hidden_view([hid[i] for i in range(nb)], m.hidden)
    seq_ids = torch.arange(Bn, dtype=torch.int32, device=dev)
    cu = (torch.arange(Bn + 1, dtype=torch.int32, device=dev) * CH).contiguous()
    for p0 in range(0, T, CH):
        for b in range(Bn):
            for i, layer in enumerate(m.band_layers):
                dt.hidden(b, layer, p0, CH, hid[i, b * CH:(b + 1) * CH], m.hidden)
        E.epikv_score_update(ctx, Bn, seq_ids, cu, CH, hv, kv)
    del hid
    torch.cuda.synchronize()
    snap = (ws.clone(), cache.k.clone(), cache.v.clone())
    kept = torch.empty((Bn, K), dtype=torch.int32, device=dev)
    nk = torch.empty(Bn, dtype=torch.int32, device=dev)
    bud = torch.full((Bn,), K, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    def restore():
        ws.copy_(snap[0])
        cache.k.copy_(snap[1])
        cache.v.copy_(snap[2])
        torch.cuda.synchronize()

    def evict():
        E.epikv_select(ctx, Bn, seq_ids, bud, None, kept, K, nk)
        E.epikv_compact(ctx, Bn, seq_ids, kept, K, kv)

    for _ in range(warmup):
        restore()
        evict()
    sel, cmp_, tot, rows = [], [], [], 0
    clocks = Clocks(Clocks.device_id(dev, local_rank)).start()
    for _ in range(steps):
        restore()
        s0 = E.epikv_get_stats(ctx)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        ev[0].record(stream)
        E.epikv_select(ctx, Bn, seq_ids, bud, None, kept, K, nk)
        ev[1].record(stream)
        E.epikv_compact(ctx, Bn, seq_ids, kept, K, kv)
        ev[2].record(stream)
        torch.cuda.synchronize()
        rows += E.epikv_get_stats(ctx)["rows_moved"] - s0["rows_moved"]
        sel.append(ev[0].elapsed_time(ev[1]))
        cmp_.append(ev[1].elapsed_time(ev[2]))
        tot.append(ev[0].elapsed_time(ev[2]))
    clk = clocks.stop()
    assert (nk.cpu().numpy() == K).all()
    peak, peak_src = measured_hbm_peak()
    restore()
    s0 = E.epikv_get_stats(ctx)
    recs = kernel_pass(E, ctx, 8, evict)
    s1 = E.epikv_get_stats(ctx)
    kernels = kernel_table(recs, 1, stream_bytes(m, tokens=0, seq_calls=0, rows_moved=s1["rows_moved"] - s0["rows_moved"],
                                                 kinds=E.EPIKV_SCORE_BANDZ, one_token=False), peak)
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code}"
    E.epikv_destroy(ctx)
    row_bytes = L * 2 * H * d * 2
    cbytes = 2 * rows / steps * row_bytes
    c_ms = float(np.median(cmp_))
    return {"workload": "batch4_64k_bandz_single_eviction_to_K4096", "steps": steps, "warmup": warmup,
            "ms_per_eviction": float(np.median(tot)), "select_ms": float(np.median(sel)), "compact_ms": c_ms,
            "candidates_per_sequence": T - 128, "rows_moved_per_eviction": rows / steps,
            "compaction_gbs": cbytes / (c_ms / 1e3) / 1e9, "compaction_frac": cbytes / (c_ms / 1e3) / 1e9 / peak,
            "peak_source": peak_src, "kernels": kernels, "clocks": clk,
            "timing": "median over evictions, each from the restored post-scoring state; CUDA events around "
                      "epikv_select and epikv_compact"}


# --------------------------------------------------------------------------- per-layer budgets
def run_layers32k(args):
    """Per-layer budgets on the 32 x 32k Lag-KV paged workload: layer l of
    every sequence keeps its own budget K_l (a pyramid from 1.5 K at layer 0
    to 0.5 K at the last layer, mean K) in its own blocks of one shared pool
    (a block table per layer), so a layer holds at most K_l + C tokens and
    the pool is sized by the budgets.  Every step evicts every layer that is
    over its budget (trigger K_min + C - 1).  One step = C new tokens per
    sequence: scoring, the per-layer selection and the per-layer compaction
    (epikv_step).  Each step's new K/V rows go to every layer's own next
    slots, which depend on the previous step, so they are written between
    steps, untimed (in a decode loop the model's forward writes them); the
    time is the sum of the steps' device times (CUDA events on the launching
    stream).  The caches are filled by the same steps, untimed."""
    import torch

    from paper_2606_26472_gb300 import epikv as E
    from paper_2606_26472_gb300.cache import KVCache
    from synth import gen, workloads as W
    from synth.device import DeviceTrace

    _, local_rank, world = dist_env()
    assert world == 1, "the per-layer budget workload is a single-GPU measurement"
    dev = gpu_device(local_rank)
    wl = W.config(3)
    m = wl.model
    Bn, K, C = args.sequences, args.budget, args.chunk
    L, H, d = m.num_layers, m.num_kv_heads, m.head_dim
    bs = wl.block_size
    budgets = W.pyramid_budgets(K, L)
    K_max, K_min = max(budgets), min(budgets)
    T_cap = K_max + C
    assert T_cap % bs == 0 and C % bs == 0 and all(k % bs == 0 for k in budgets)
    mb = T_cap // bs
    need = [(k + C) // bs for k in budgets]           # blocks a layer of a sequence ever holds
    n_blocks = Bn * sum(need)
    perm = gen.block_permutation(m.seed, n_blocks)
    tab = np.full((L, Bn, mb), -1, np.int32)
    o = 0
    for l in range(L):
        for b in range(Bn):
            tab[l, b, :need[l]] = perm[o:o + need[l]]
            o += need[l]
    cache = KVCache(E.EPIKV_LAYOUT_PAGED, L, H, d, max_seqs=Bn, max_tokens=T_cap, block_size=bs,
                    num_blocks=n_blocks, block_table=tab, layer_tables=True, device=dev)
    view = cache.view()
    stage = KVCache(E.EPIKV_LAYOUT_CONTIGUOUS, L, H, d, max_seqs=Bn, max_tokens=C, device=dev)
    dt = DeviceTrace(m, dev)
    stream = torch.cuda.current_stream()
    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=T_cap, max_new_tokens=C, num_layers=L, num_kv_heads=H,
                        head_dim=d, lag=wl.lag, lag_window=wl.lag_window, recency_cap=wl.recency_cap,
                        score_kinds=E.EPIKV_SCORE_LAGKV, layer_budgets=1)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device=dev)
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, E.EPIKV_SCORE_LAGKV)
    seq_ids = torch.arange(Bn, dtype=torch.int32, device=dev)
    cu_new = (torch.arange(Bn + 1, dtype=torch.int32, device=dev) * C).contiguous()
    budget = torch.tensor([list(budgets)] * Bn, dtype=torch.int32, device=dev)
    trigger = torch.full((Bn,), K_min + C - 1, dtype=torch.int32, device=dev)
    n_out = torch.empty((Bn, L), dtype=torch.int32, device=dev)
    n_layer = np.zeros((Bn, L), dtype=np.int64)
    rows = np.arange(Bn)[:, None]

    def write_new(pos0):   # step's new rows into every layer's next C slots
        for b in range(Bn):
            dt.kv(b, pos0, C, 0, stage.k, stage.v, **dict(stage.synth_kwargs(), stride_seq=C * H * d))
        for l in range(L):
            slots = n_layer[:, l:l + 1] + np.arange(C)
            flat = tab[l][rows, slots // bs] * bs + slots % bs
            idx = torch.as_tensor(flat.reshape(-1), device=dev)
            cache.k.view(-1, H, d)[idx] = stage.k[l].reshape(-1, H, d)
            cache.v.view(-1, H, d)[idx] = stage.v[l].reshape(-1, H, d)

    fill = K_max // C                                   # steps until every layer has reached its budget
    n_steps = fill + args.warmup + args.steps
    t0 = fill + args.warmup
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_steps)]
    phase = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_steps)]
    for e in (x for p in phase for x in p):
        e.record(stream)   # materialise the handles
    gpu_id = Clocks.device_id(dev, local_rank)
    clocks = None
    stats0 = None
    for st in range(n_steps):
        if st == t0:
            torch.cuda.synchronize()
            stats0 = E.epikv_get_stats(ctx)
            clocks = Clocks(gpu_id).start()
        write_new(st * C)
        E.epikv_set_phase_events(ctx, phase[st])
        ev[st][0].record(stream)
        E.epikv_step(ctx, Bn, seq_ids, cu_new, C, budget, trigger, None, view, n_out)
        ev[st][1].record(stream)
        n_layer = n_out.cpu().numpy().astype(np.int64)
        assert (n_layer <= np.asarray(budgets)[None, :] + C).all()
    torch.cuda.synchronize()
    clk = clocks.stop()
    E.epikv_set_phase_events(ctx, None)
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code}"
    assert (n_layer == np.asarray(budgets)[None, :]).all()
    stats1 = E.epikv_get_stats(ctx)
    timed = range(t0, n_steps)
    ms = sum(ev[i][0].elapsed_time(ev[i][1]) for i in timed)
    t_score = sum(phase[i][0].elapsed_time(phase[i][1]) for i in timed)
    t_select = sum(phase[i][1].elapsed_time(phase[i][2]) for i in timed)
    t_compact = sum(phase[i][2].elapsed_time(phase[i][3]) for i in timed)
    tokens = stats1["tokens_scored"] - stats0["tokens_scored"]
    assert tokens == Bn * C * args.steps
    layer_rows = stats1["layer_rows_moved"] - stats0["layer_rows_moved"]
    compact_bytes = 2 * layer_rows * 2 * H * d * 2          # read + write of K and V rows of one layer
    peak, peak_src = measured_hbm_peak()
    ach = compact_bytes / (t_compact / 1e3) / 1e9
    block_bytes = 2 * bs * H * d * 2                        # K and V of one block
    E.epikv_destroy(ctx)
    return {
        "metric": METRIC, "value": tokens / (ms / 1e3), "unit": UNIT, "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": f"batch{Bn}_32k_lagkv_paged16_layerbudgets_pyramid_mean{K}_chunk{C}",
                   "sequences": Bn, "layers": L, "kv_heads": H, "head_dim": d, "chunk": C,
                   "layer_budgets": [budgets[0], budgets[-1]], "budget_mean": K, "score": "lagkv_lag16_w64",
                   "pool": "one block pool, a block table per layer: %.1f GiB (one table for all layers: %.1f GiB)"
                           % (n_blocks * block_bytes / 2 ** 30, Bn * mb * L * block_bytes / 2 ** 30),
                   "timing": "sum of per-step device times; each step's new K/V written before it, untimed",
                   "l2": "inputs larger than L2"},
        "kernels_ms_per_step": {"score": t_score / args.steps, "select": t_select / args.steps,
                                "compact": t_compact / args.steps},
        "roofline": {"bound": "hbm", "kernel": "compact_kernel", "achieved": ach, "peak": peak, "unit": "GB/s",
                     "frac": ach / peak, "peak_source": peak_src, "traffic": None,
                     "algorithmic_bytes_per_launch": compact_bytes / args.steps},
        # Lag-KV partial, finalize, layer keep, layer union, [stash: at most 256 (sequence, layer)
        # pairs,] compaction, consumed
        "gpu_launches": (7 if Bn * L <= 256 else 6) * args.steps,
        "clocks": clk,
    }


# --------------------------------------------------------------------------- configurations 2 and 5
def window_schedule(n0, budgets, slack, C, n_calls):
    """The decode window's rows, simulated on the host: per call, every
    sequence's C new tokens (positions continuing from n0, slots from its
    cache length), and the sequences that evict (cache length > K + slack,
    cut back to K).  Returns (positions [n_calls][B*C], slots [n_calls][B*C],
    evictions per call, cache lengths after the last call)."""
    B = len(n0)
    n_cache = np.array(n0, dtype=np.int64)
    budgets = np.asarray(budgets, dtype=np.int64)
    pos_tab = np.empty((n_calls, B * C), np.int32)
    slot_tab = np.empty((n_calls, B * C), np.int32)
    evict_tab = np.zeros(n_calls, np.int64)
    r = np.arange(C)
    for j in range(n_calls):
        pos_tab[j] = (np.asarray(n0)[:, None] + j * C + r[None, :]).reshape(-1)
        slot_tab[j] = (n_cache[:, None] + r[None, :]).reshape(-1)
        n_cache += C
        ev = n_cache > budgets + slack
        evict_tab[j] = int(ev.sum())
        n_cache[ev] = budgets[ev]
    return pos_tab, slot_tab, evict_tab, n_cache


def run_window(args, workload=None, steps=None, warmup=None):
    """Steady-state decode windows of two more workloads, timed per
    epikv_step call with CUDA events on the stream; the generator kernels
    that append each call's new rows (the model's side of the loop) run
    between the events:
    * bandz8k (configuration 2): 8 x 8,192-token band-z traces, contiguous
      K/V, K = 4,096; 64 new tokens per sequence per call, every call evicts
      back to K;
    * ragged64 (configuration 5): 64 sequences with budgets from {2048,
      4096, 8192}, paged 16-token blocks, both scores, one new token per
      sequence per call; a sequence evicts when its cache exceeds K + 64.
      The sequences start at staggered lengths K + (29 b mod 65), so one of
      them evicts at nearly every call.
    One bench step = the calls in which every sequence evicts once (1 and
    65).  Every call has the same arguments, so one captured CUDA graph of
    the call is replayed; the eager rate (with the per-phase breakdown) is
    reported beside it."""
    import torch

    from paper_2606_26472_gb300 import epikv as E
    from paper_2606_26472_gb300.cache import KVCache
    from synth import gen, workloads as W
    from synth.device import DeviceBatchTrace

    _, local_rank, world = dist_env()
    assert world == 1, "the decode-window workloads are single-GPU measurements"
    dev = gpu_device(local_rank)
    workload = workload or args.workload
    steps = args.steps if steps is None else steps
    warmup = args.warmup if warmup is None else warmup
    ragged = workload == "ragged64"
    wl = W.config(5 if ragged else 2)
    scaled = bool(args.window_seqs or args.window_budget)
    if scaled:
        import dataclasses
        n_keep = args.window_seqs or wl.n_seq
        bud = (args.window_budget,) * n_keep if args.window_budget else wl.budgets[:n_keep]
        wl = dataclasses.replace(wl, n_seq=n_keep, lengths=wl.lengths[:n_keep], budgets=bud,
                                 policies=wl.policies[:n_keep], trigger_slack=wl.trigger_slack[:n_keep])
    m = wl.model
    L, H, d, nb = m.num_layers, m.num_kv_heads, m.head_dim, len(m.band_layers)
    Bn, C = wl.n_seq, wl.chunk
    budgets = np.array(wl.budgets, dtype=np.int64)
    slack = wl.trigger_slack[0]
    assert all(s == slack for s in wl.trigger_slack)
    cycle = slack + 1                   # new tokens of a sequence between two of its evictions
    calls = cycle // C                  # calls per bench step
    assert calls * C == cycle
    phase0 = (np.arange(Bn) * 29) % cycle if C == 1 else np.zeros(Bn, np.int64)
    n0 = budgets + phase0
    T_cap = int(budgets.max()) + cycle
    kc_calls = calls if ragged else 3   # the per-kernel pass: one step of 65 calls, or 3 calls
    n_calls = 2 * (warmup + steps) * calls + kc_calls     # eager run, graph run, per-kernel pass
    max_pos = int(n0.max()) + n_calls * C + 1
    paged = wl.layout == W.PAGED
    if paged:
        mb = (T_cap + wl.block_size - 1) // wl.block_size
        bt = gen.block_permutation(m.seed, Bn * mb).reshape(Bn, mb)
        cache = KVCache(E.EPIKV_LAYOUT_PAGED, L, H, d, max_seqs=Bn, max_tokens=T_cap, block_size=wl.block_size,
                        block_table=bt, device=dev)
    else:
        cache = KVCache(E.EPIKV_LAYOUT_CONTIGUOUS, L, H, d, max_seqs=Bn, max_tokens=T_cap, device=dev)
    kv = cache.view()
    setup_chunk = 256
    cfg = E.make_config(max_seqs=Bn, max_cache_tokens=T_cap, max_new_tokens=max(setup_chunk, C), num_layers=L,
                        num_kv_heads=H, head_dim=d, hidden=m.hidden, n_band_a=len(m.band_a),
                        n_band_b=len(m.band_b), z_window=wl.z_window, lag=wl.lag, lag_window=wl.lag_window,
                        recency_cap=wl.recency_cap, score_kinds=wl.kinds)
    ws = torch.empty(E.epikv_workspace_bytes(cfg), dtype=torch.uint8, device=dev)
    ctx = E.epikv_init(cfg, ws, ws.numel())
    for b in range(Bn):
        E.epikv_seq_reset(ctx, b, 0, wl.policies[b])
    dt = DeviceBatchTrace(m, Bn, max_pos, dev)

    # every sequence's first n0 tokens, scored in chunks (no eviction yet)
    hs = torch.empty((nb, setup_chunk, m.hidden), dtype=torch.bfloat16, device=dev)
    hv_s = E.hidden_view([hs[i] for i in range(nb)], m.hidden)
    cu_s = {}
    for b in range(Bn):
        ids = torch.tensor([b], dtype=torch.int32, device=dev)
        for p0 in range(0, int(n0[b]), setup_chunk):
            c = min(setup_chunk, int(n0[b]) - p0)
            if c not in cu_s:
                cu_s[c] = torch.tensor([0, c], dtype=torch.int32, device=dev)
            for i, layer in enumerate(m.band_layers):
                dt.hidden(b, layer, p0, c, hs[i], m.hidden)
            dt.kv(b, p0, c, p0, cache.k, cache.v, **cache.synth_kwargs())
            E.epikv_score_update(ctx, 1, ids, cu_s[c], c, hv_s, kv)

    pos_tab, slot_tab, evict_tab, n_cache = window_schedule(n0, budgets, slack, C, n_calls)
    seq_rows = torch.from_numpy(np.repeat(np.arange(Bn, dtype=np.int32), C)).to(dev)
    pos_dev = torch.from_numpy(pos_tab).to(dev)
    slot_dev = torch.from_numpy(slot_tab).to(dev)
    hid = torch.empty((nb, Bn * C, m.hidden), dtype=torch.bfloat16, device=dev)
    hv = E.hidden_view([hid[i] for i in range(nb)], m.hidden)
    seq_ids = torch.arange(Bn, dtype=torch.int32, device=dev)
    cu = (torch.arange(Bn + 1, dtype=torch.int32, device=dev) * C).contiguous()
    bud = torch.from_numpy(budgets.astype(np.int32)).to(dev)
    trig = (bud + slack).contiguous()
    n_out = torch.empty(Bn, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code} during set-up"

    def append(j):   # call j's new rows: hidden rows of the band layers, K/V into their slots
        for i, layer in enumerate(m.band_layers):
            dt.hidden_batch(layer, seq_rows, pos_dev[j], hid[i], m.hidden)
        dt.kv_batch(seq_rows, pos_dev[j], slot_dev[j], cache.k, cache.v, **cache.synth_kwargs())

    def call():
        E.epikv_step(ctx, Bn, seq_ids, cu, C, bud, trig, hv, kv, n_out)

    j = 0

    def window(n_steps, run, timed, phases=False):
        nonlocal j
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n_steps * calls)] if timed else []
        ph = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_steps * calls)] \
            if phases else []
        for p in ph:
            for e in p:
                e.record(stream)   # materialise the handles
        for k in range(n_steps * calls):
            append(j)
            if ph:
                E.epikv_set_phase_events(ctx, ph[k])
            if ev:
                # ~0.1 ms of device spin ahead of the start event: the whole
                # call is queued before the device reaches it, so no host
                # submission gap falls between the events
                torch.cuda._sleep(200000)
                ev[k][0].record(stream)
            run()
            if ev:
                ev[k][1].record(stream)
            j += 1
        torch.cuda.synchronize()
        E.epikv_set_phase_events(ctx, None)
        ms = sum(a.elapsed_time(b_) for a, b_ in ev)
        per_phase = [sum(p[q].elapsed_time(p[q + 1]) for p in ph) for q in range(3)] if ph else None
        return ms, per_phase

    gpu_id = Clocks.device_id(dev, local_rank)
    window(warmup, call, False)
    s0 = E.epikv_get_stats(ctx)
    j0 = j
    ms_eager, (t_score, t_select, t_compact) = window(steps, call, True, phases=True)
    s1 = E.epikv_get_stats(ctx)
    assert s1["evictions"] - s0["evictions"] == int(evict_tab[j0:j].sum())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        call()
    window(warmup, g.replay, False)
    clocks = Clocks(gpu_id).start()
    s2 = E.epikv_get_stats(ctx)
    j2 = j
    ms_graph, _ = window(steps, g.replay, True)
    clk = clocks.stop()
    s3 = E.epikv_get_stats(ctx)
    assert s3["evictions"] - s2["evictions"] == int(evict_tab[j2:j].sum())
    # per-kernel CUDA events over kc_calls eager calls
    peak, peak_src = measured_hbm_peak()

    def kc_run():
        nonlocal j
        for _ in range(kc_calls):
            append(j)
            call()
            j += 1

    s4 = E.epikv_get_stats(ctx)
    recs = kernel_pass(E, ctx, 8 * kc_calls, kc_run)
    s5 = E.epikv_get_stats(ctx)
    assert j == n_calls
    kernels = kernel_table(recs, kc_calls / calls,
                           stream_bytes(m, tokens=kc_calls * Bn * C, seq_calls=kc_calls * Bn,
                                        rows_moved=s5["rows_moved"] - s4["rows_moved"], kinds=wl.kinds,
                                        one_token=C == 1), peak)
    st_, code = E.epikv_get_error(ctx)
    assert st_ == E.EPIKV_OK, f"device error {code}"
    for b in range(Bn):   # the device's cache lengths follow the host's simulation
        _, _, n = E.epikv_read_slots(ctx, b, wl.policies[b], 1)
        assert n == n_cache[b], (b, n, int(n_cache[b]))
    E.epikv_destroy(ctx)

    tokens = steps * calls * Bn * C
    assert s3["tokens_scored"] - s2["tokens_scored"] == tokens
    row_bytes = L * 2 * H * d * 2
    rows = s1["rows_moved"] - s0["rows_moved"]
    compact_bytes = 2 * rows * row_bytes
    n_launch = calls * steps
    ach = compact_bytes / (t_compact / 1e3) / 1e9
    name = ("ragged64_4k32k_both_paged16_steady" if ragged else "batch8_8k_bandz_contiguous_K4096_every64")
    if scaled:
        name += f"_first{Bn}seqs" + (f"_K{args.window_budget}" if args.window_budget else "")
    return {"metric": METRIC, "value": tokens / (ms_graph / 1e3), "unit": UNIT, "n_gpus": 1,
            "steps": steps, "warmup": warmup, "ms_per_step": ms_graph / steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": name, "sequences": Bn, "budgets": sorted(set(wl.budgets)),
                       "new_tokens_per_call": C, "calls_per_step": calls,
                       "evict_when": f"n_cache > K + {slack}", "layout": "paged16_shuffled" if paged else "contiguous",
                       "score_kinds": wl.kinds, "timing": "CUDA events around each epikv_step call, queued behind a device spin",
                       "l2": "K/V caches %.1f GiB, larger than L2" % (cache.k.numel() * 4 / 2 ** 30)},
            "eager_value": tokens / (ms_eager / 1e3),
            "us_per_call": {"graph": 1e3 * ms_graph / n_launch, "eager": 1e3 * ms_eager / n_launch},
            "kernels_ms_per_step": {"score": t_score / steps, "select": t_select / steps,
                                    "compact": t_compact / steps},
            "evictions_per_step": (s1["evictions"] - s0["evictions"]) / steps,
            "compaction_gbs": ach, "compaction_frac": ach / peak,
            "roofline": {"bound": "hbm", "kernel": "compact_kernel", "achieved": ach, "peak": peak, "unit": "GB/s",
                         "frac": ach / peak, "peak_source": peak_src, "traffic": None,
                         "algorithmic_bytes_per_launch": compact_bytes / n_launch,
                         "timing": "eager calls, phase events"},
            "kernels": kernels,
            # one-token calls: the fused score kernel, select, stash, compaction, eviction
            # consumed; longer calls: g, [Lag-KV partial,] finalize and the same four
            "gpu_launches": (5 if C == 1 else (7 if wl.kinds & E.EPIKV_SCORE_LAGKV else 6)) * n_launch,
            "clocks": clk}


# --------------------------------------------------------------------------- the per-configuration table
def _entry(res, step):
    keys = ("value", "unit", "ms_per_step", "steps", "warmup", "compaction_gbs", "compaction_frac",
            "kernels_ms_per_step", "kernels", "clocks")
    out = {"workload": res["config"]["workload"], "step": step}
    out.update({k: res[k] for k in keys if k in res})
    return out


def collect_configs(args, headline):
    """Every workload measured one after another on this GPU (each with its
    own clocks record and per-kernel CUDA-event pass), reduced step counts."""
    import gc

    import torch

    def free():
        gc.collect()
        torch.cuda.empty_cache()

    t0 = time.time()
    out = {}
    free()
    r = run_bandz2k(args, steps=10, warmup=3)
    out["1"] = _entry(r, "one fresh sequence: 2,048 tokens scored (band-z), one eviction 2,048 -> 512")
    out["1"]["score_phase_gbs"] = r["score_phase_gbs"]
    free()
    r = run_window(args, "bandz8k", steps=20, warmup=3)
    out["2"] = _entry(r, "one epikv_step call (CUDA graph): 64 new tokens of each of 8 sequences scored (band-z), "
                         "every cache 4,160 -> 4,096")
    out["2"]["eager_value"] = r["eager_value"]
    h = headline
    out["3"] = {"workload": h["config"]["workload"], "step": "one epikv_step: 128 new tokens of each of 32 "
                "sequences scored (Lag-KV), every cache 8,320 -> 8,192", "value": h["value"], "unit": h["unit"],
                "ms_per_step": h["ms_per_step"], "steps": h["steps"], "warmup": h["warmup"],
                "compaction_gbs": h["compaction_gbs"], "compaction_frac": h["roofline"]["frac"],
                "kernels_ms_per_step": h["kernels_ms_per_step"], "kernels": h["kernels"], "clocks": h["clocks"],
                "note": "the headline measurement of this line"}
    free()
    r4a = run_pertoken(args, steps=10, warmup=3)
    free()
    r4b = run_evict64k(args, steps=3, warmup=1)
    free()
    per_step_ms = r4a["ms_per_step"] / 64          # one decode step of the 4 sequences (graph replay)
    whole_ms = 65536 * per_step_ms + r4b["ms_per_eviction"]
    out["4"] = {"workload": "batch4_64k_bandz_K4096", "step": "per-token phase: 64 decode steps of 4 sequences "
                "(one CUDA graph of 64 score updates); eviction phase: 4 x 65,536 -> 4,096",
                "per_token_phase": _entry(r4a, "64 decode steps (4 tokens each)"),
                "eviction_phase": r4b,
                "whole_schedule_tokens_per_s": 4 * 65536 / (whole_ms / 1e3),
                "whole_schedule_note": "4 x 65,536 tokens over 65,536 x the measured decode-step time plus the "
                                       "measured eviction (the phases are measured apart)"}
    r = run_window(args, "ragged64", steps=3, warmup=2)
    free()
    out["5"] = _entry(r, "65 epikv_step calls (CUDA graph), one new token of each of 64 sequences per call "
                         "(both scores); every sequence evicts once")
    out["5"]["us_per_call"] = r["us_per_call"]
    out["5"]["eager_value"] = r["eager_value"]
    out["seconds"] = time.time() - t0
    return out


def main(argv=None):
    args = parse(argv)
    if args.impl == "reference":
        run_reference(args)
        return
    if args.workload == "lagkv32k":
        line = run_ours(args)
        if line is None:
            return
        _, _, world = dist_env()
        default = line["config"]["workload"] == WORKLOAD
        if world == 1 and default and not args.no_configs:
            line["configs"] = collect_configs(args, line)
        if world == 1 and default and not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(args.cpu_workers)
        print(json.dumps(line), flush=True)
        return
    run = {"bandz2k": run_bandz2k, "pertoken": run_pertoken, "evict64k": run_evict64k, "layers32k": run_layers32k,
           "bandz8k": run_window, "ragged64": run_window}[args.workload]
    print(json.dumps(run(args)), flush=True)


if __name__ == "__main__":
    main()
