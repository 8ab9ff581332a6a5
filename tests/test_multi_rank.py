"""The multi-GPU path of bench.py on the CPU: independent replicas (the stack
does not shard), timed by the slowest rank.  Two gloo ranks on 127.0.0.1 check
that every rank sees the maximum of the per-rank times and the whole-job
throughput formula; no GPU is used."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, times, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, _ = bench.dist_env()
        slowest = bench.max_over_ranks(times[r], w, "cpu")
        q.put((r, slowest, bench.replica_throughput(w, 100, slowest)))
    finally:
        dist.barrier()
        dist.destroy_process_group()


def test_replicas_take_the_slowest_rank_gloo():
    world, port = 2, _free_port()
    times = [170.0, 212.5]  # ms of 100 steps on each rank
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, times, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for r, slowest, value in got:
        assert slowest == pytest.approx(212.5)
        assert value == pytest.approx(2 * 100 / 0.2125)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.replica_throughput(1, 2000, 3340.0) == pytest.approx(2000 / 3.34)
