"""The benchmark's multi-rank aggregation on two gloo ranks (CPU): every rank
runs its own replica; the barrier and the max over ranks of the step time
follow the launch contract (torchrun, one process per GPU)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # rank r measured (r + 1) ms; the job's time is the slowest rank's
    v = bench._max_over_ranks(1.0 + rank, world, torch.device("cpu"))
    bench._barrier(world)
    q.put((rank, v))
    dist.destroy_process_group()


def test_max_over_ranks_and_barrier_gloo():
    ctx = torch.multiprocessing.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert out == {0: 2.0, 1: 2.0}


def test_single_rank_needs_no_process_group():
    import bench
    assert bench._max_over_ranks(3.5, 1, None) == 3.5
    bench._barrier(1)
