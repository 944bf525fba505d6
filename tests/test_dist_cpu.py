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


# ---- number-wise partitioned table (App. D): the exchange on CPU ----------

class _NumpySteps:
    """The local steps of one rank in plain numpy (test infrastructure): the
    exchange and re-assembly of paper_2411_12364_gb300.shard are checked with
    them; the library's kernels for the same steps are checked on a GPU."""

    def __init__(self, cfg, t, lo, hi):
        import numpy as np
        self.np = np
        self.cfg, self.t = cfg, t
        self.shard = t["values"][lo:hi]
        self.N = int(cfg["n"]) ** 2

    def _rows(self, idx):
        import oracle
        v = oracle.shuffle(self.cfg, idx.numpy())
        return v // self.N, v % self.N

    def route(self, idx, P, R):
        import torch
        np = self.np
        _, row = self._rows(idx)
        row = row.ravel()
        owner = row // R
        order = np.argsort(owner, kind="stable")
        counts = np.bincount(owner, minlength=P).astype(np.int32)
        slot_pos = np.empty(row.size, np.int32)
        slot_pos[order] = np.arange(row.size, dtype=np.int32)
        send = (row - owner * R)[order].astype(np.int32)
        return torch.from_numpy(counts), torch.from_numpy(send), torch.from_numpy(slot_pos)

    def lookup(self, rows):
        import torch
        return torch.from_numpy(self.shard[rows.numpy()].astype(self.np.float32))

    def pool(self, idx, w, slot_pos, rows):
        import torch
        np = self.np
        blk, _ = self._rows(idx)
        n, E, dv = idx.shape[0], int(self.cfg["expand_e"]), int(self.cfg["d_v"])
        blk = blk.reshape(n, -1)
        ww = w.numpy().astype(np.float64).reshape(n, -1)
        back = rows.numpy().astype(np.float64)
        pos = slot_pos.numpy().reshape(n, -1)
        acc = np.zeros((n, E, dv))
        for b in range(n):
            for s in range(blk.shape[1]):
                acc[b, blk[b, s]] += ww[b, s] * back[pos[b, s]]
        wp = np.asarray(self.t["w_proj"], np.float64).reshape(E, dv, -1)
        return torch.from_numpy(np.einsum("bpc,pco->bo", acc, wp))


def _shard_worker(rank, world, port, queue):
    import sys
    import numpy as np
    import torch
    import torch.distributed as dist
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from paper_2411_12364_gb300 import shard, workloads
    cfg = workloads.small_config(dtype=0, n=11)            # N = 121 rows: shards of 61 and 60
    w = workloads.make_weights(cfg, device="cpu")
    t = {k: workloads.stored_numpy(v) for k, v in w.items() if k in ("values", "w_proj")}
    N = int(cfg["n"]) ** 2
    lo, hi = shard.shard_bounds(N, world, rank)
    table = shard.NumberWiseTable(_NumpySteps(cfg, t, lo, hi), N, cfg["d_v"])
    gen = torch.Generator().manual_seed(100 + rank)
    n, M = 5 + rank, int(cfg["expand_e"]) * N
    idx = torch.randint(0, M, (n, cfg["heads"], cfg["topm"]), generator=gen)
    wt = torch.randn((n, cfg["heads"], cfg["topm"]), generator=gen)
    out = table.lookup_reduce(idx, wt).numpy()
    want = oracle.lookup_reduce(cfg, t, idx.numpy(), wt.numpy().astype(np.float64))
    err = float(np.abs(out - want).max() / np.abs(want).max())
    queue.put((rank, err, table.last, hi - lo))
    dist.barrier()
    dist.destroy_process_group()


def test_number_wise_table_exchange_two_ranks():
    """Each rank holds half the rows, routes its own slots to the owners,
    serves the rows requested from it and pools what comes back: its output
    is the oracle's lookup-reduce over the whole table."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    results = sorted(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    served = 0
    for rank, err, last, rows in results:
        assert err <= 1e-12, f"rank {rank}: {err}"
        assert rows == (61 if rank == 0 else 60)
        assert last["slots"] == (5 + rank) * 2 * 8
        assert 0 < last["index_bytes_sent"] < 4 * last["slots"]
        served += last["requests_served"]
    assert served == sum(r[2]["slots"] for r in results)   # every request answered once
