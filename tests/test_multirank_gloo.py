"""The N-replica aggregation of bench.py on two CPU ranks (gloo): the whole-job
value is every rank's work over the slowest rank's time."""
import os
import socket

import pytest
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

    flops, secs = bench.aggregate(1e12 * (rank + 1), 0.5 + rank, world)
    q.put((rank, flops, secs))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_aggregate():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for _, flops, secs in out:
        assert flops == pytest.approx(3e12) and secs == pytest.approx(1.5)


def test_single_rank_is_identity():
    import bench

    assert bench.aggregate(5.0, 2.0, 1) == (5.0, 2.0)
