"""Multi-rank bench plumbing on CPU (gloo, world size 2): each rank runs its
own replica on its own batch; the reported step time is the slowest rank's
and the throughput counts every rank's tokens."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, queue):
    import sys
    import torch.distributed as dist
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, value = bench.aggregate_step(1.5 + rank, 64, dist)
    queue.put((rank, ms, value))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_max_time_and_total_tokens():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    results = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, value in results:
        assert ms == pytest.approx(2.5)                 # the slower rank
        assert value == pytest.approx(2 * 64 / 2.5e-3)  # both ranks' tokens


def test_single_process_aggregation():
    import bench
    ms, value = bench.aggregate_step(2.0, 64)
    assert ms == 2.0 and value == pytest.approx(32000.0)
