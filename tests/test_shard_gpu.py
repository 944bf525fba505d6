"""The local steps of the number-wise partitioned table (App. D) on one GPU:
two ranks' shards of the table, each behind its own layer, are served in
one process and the exchanges are done by slicing (no kernel waits on
another).  Each rank's output must be the oracle's lookup-reduce over the
whole table, and bit-identical to the unpartitioned layer's lookup-reduce
of the same slots."""
import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import binding, shard, workloads
from tests import parity

pytestmark = pytest.mark.gpu


def _exchange(sends, counts, P):
    """recv[o]: what the P ranks send to owner o, in rank order; and where
    each rank's block for each owner starts."""
    starts = [np.concatenate([[0], np.cumsum(c)]) for c in counts]
    recv = [torch.cat([sends[q][starts[q][o]:starts[q][o + 1]] for q in range(P)])
            for o in range(P)]
    return recv, starts


@pytest.mark.parametrize("name,B,cores", [("decode_1m", 64, 0), ("tiny_fp32", 16, 0),
                                          ("decode_1m", 32, 2)])
def test_number_wise_local_steps(name, B, cores, gpu_lib):
    cfg = workloads.layer_config(name, cores=cores)
    w = workloads.make_weights(cfg, device="cuda")
    N = int(cfg["n"]) ** 2
    P = 2
    R = shard.rows_per_rank(N, P)
    full = binding.UltraMemLayer(cfg, w, B)
    layers, idxs, wts = [], [], []
    for q in range(P):
        lo, hi = shard.shard_bounds(N, P, q)
        lw = dict(w, values=w["values"][lo:hi])
        layers.append(binding.UltraMemLayer(dict(cfg, shard_rows=hi - lo), lw, B))
        x = workloads.make_tokens(cfg, B, batch_index=q, device="cuda")
        i, wt = layers[q].retrieve(x)
        if q == 1:
            i[2, 0, 1] = int(cfg["expand_e"]) * N + 3   # outside the grid: skipped
        idxs.append(i)
        wts.append(wt)
    with pytest.raises(binding.UltraMemError):
        layers[0].forward(workloads.make_tokens(cfg, B, device="cuda"))
    routed = [layers[q].shard_route(idxs[q], P, R) for q in range(P)]
    counts = [r[0].cpu().numpy() for r in routed]
    assert all(c.sum() == idxs[q].numel() for q, c in enumerate(counts))
    recv, starts = _exchange([r[1] for r in routed], counts, P)
    served = [layers[o].shard_lookup(recv[o]) for o in range(P)]
    # rows back: owner o's answer to rank q follows the ranks before q
    t = {k: workloads.stored_numpy(v) for k, v in w.items() if k in ("values", "w_proj")}
    for q in range(P):
        parts = []
        for o in range(P):
            before = sum(int(counts[r][o]) for r in range(q))
            parts.append(served[o][before:before + int(counts[q][o])])
        back = torch.cat(parts)
        out = layers[q].shard_pool(idxs[q], wts[q], routed[q][2], back)
        torch.cuda.synchronize()
        i_np = idxs[q].cpu().numpy().copy()
        w_np = wts[q].cpu().numpy().astype(np.float64).copy()
        bad = (i_np < 0) | (i_np >= int(cfg["expand_e"]) * N)
        i_np[bad] = 0
        w_np[bad] = 0.0
        want = oracle.lookup_reduce(cfg, t, i_np, w_np)
        err, _ = parity.output_errors(out.float().cpu().numpy(), want)
        assert err.max() <= parity.out_tol(cfg), f"rank {q}: {err.max()}"
        ref = full.lookup_reduce(idxs[q], wts[q])
        assert torch.equal(out, ref), f"rank {q} differs from the unpartitioned lookup"
    assert layers[1].check() == binding.EDEVICE    # the out-of-grid address was recorded
    for L in layers + [full]:
        L.close()


def test_shard_lookup_rejects_rows_outside_its_shard(gpu_lib):
    cfg = workloads.small_config(dtype=1, n=10)
    w = workloads.make_weights(cfg, device="cuda")
    layer = binding.UltraMemLayer(dict(cfg, shard_rows=30), dict(w, values=w["values"][:30]), 4)
    rows = torch.tensor([0, 29, 30, -1], dtype=torch.int32, device="cuda")
    out = layer.shard_lookup(rows)
    torch.cuda.synchronize()
    assert torch.equal(out[0], w["values"][0]) and torch.equal(out[1], w["values"][29])
    assert (out[2:] == 0).all()
    assert layer.check() == binding.EDEVICE
    layer.close()
