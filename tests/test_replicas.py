"""Multi-process (world size 2, gloo, CPU) check of the benchmark's replica
aggregation: every rank runs an independent replica; the reported value is all
ranks' units over the slowest rank's time. No GPU, no data-path collective."""
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
    try:
        import bench

        local_ms = [1000.0, 1500.0][rank]  # rank 1 is the slow replica
        value, ms_max = bench.replica_throughput(local_ms, units_per_step=3e9, steps=4, world=world,
                                                 device=torch.device("cpu"))
        q.put((rank, value, ms_max))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_replica_throughput_two_ranks_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, value, ms_max in got:
        assert ms_max == 1500.0
        assert value == pytest.approx(2 * 4 * 3e9 / 1.5)


def test_replica_throughput_single_process():
    import bench

    value, ms_max = bench.replica_throughput(250.0, 1e9, 2, 1, torch.device("cpu"))
    assert ms_max == 250.0 and value == pytest.approx(8e9)
