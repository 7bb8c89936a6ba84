"""The N > 1 host logic on CPU: world-size-2 gloo ranks (no GPU).

The eviction path shards by sequence (every rank owns whole sequences and
their KV), so ranks never exchange data; only the bench's timing needs the
ranks: the job's duration is the slowest rank's, and the throughput counts
every rank's tokens once.
"""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms, value = bench.aggregate_ranks(10.0 * (rank + 1), 4096, world)
    q.put((rank, ms, value))
    dist.barrier()
    dist.destroy_process_group()


def test_weak_scaling_aggregation_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, ms, value in got:
        assert ms == 20.0                       # the slowest rank's time
        assert value == pytest.approx(2 * 4096 / 0.020)   # all ranks' tokens over it


def _shard_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    mine = bench.shard_sequences(32, rank, world)
    owned = [None] * world
    dist.all_gather_object(owned, mine)
    tokens = 128 * len(mine) * (rank + 1)          # ranks may process different amounts
    ms, value = bench.aggregate_ranks(5.0 + rank, tokens, world)
    q.put((rank, owned, ms, value))
    dist.barrier()
    dist.destroy_process_group()


def test_sequence_sharding_over_two_gloo_ranks():
    """Every global sequence is owned by exactly one rank, and the job's
    throughput counts each rank's tokens once over the slowest rank's time."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, owned, ms, value in got:
        flat = [s for o in owned for s in o]
        assert sorted(flat) == list(range(64)) and len(set(flat)) == 64   # disjoint, covers the global batch
        assert owned[rank] == list(range(32 * rank, 32 * rank + 32))
        assert ms == 6.0
        assert value == pytest.approx((128 * 32 * 1 + 128 * 32 * 2) / 0.006)
    # one rank owning the whole batch counts the same tokens
    import bench
    assert bench.shard_sequences(64, 0, 1) == list(range(64))


def test_single_rank_aggregation_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_ranks(8.0, 1000, 1) == (8.0, 1000 / 0.008)


def test_reference_arm_runs_on_rank_zero_only(capsys, monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = type("A", (), {"steps": 1, "warmup": 1, "gpus": 2})()
    assert bench.run_reference(args) is None
    assert capsys.readouterr().out == ""
