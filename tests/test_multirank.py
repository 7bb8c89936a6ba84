"""The N > 1 host logic on CPU: world-size-2 gloo ranks (no GPU).

The eviction path shards by sequence (every rank owns whole sequences and
their KV), so ranks never exchange data; only the bench's timing needs the
ranks: the job's duration is the slowest rank's, and the throughput counts
every rank's tokens.
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
