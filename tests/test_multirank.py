"""Multi-rank host logic of bench.py (replicas, max over ranks) on two gloo
ranks on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    step_ms = [1.5, 2.5][rank]
    value, t = bench.aggregate(step_ms, 64, world, dist, "cpu")
    dist.barrier()
    q.put((rank, value, t))
    dist.destroy_process_group()


def test_two_rank_aggregate_is_max_over_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, value, t in res:
        assert t == pytest.approx(2.5)
        assert value == pytest.approx(2 * 64 / 2.5e-3)


def test_single_rank_aggregate():
    import bench
    value, t = bench.aggregate(2.0, 64, 1)
    assert t == 2.0 and value == pytest.approx(32000.0)
