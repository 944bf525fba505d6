"""Number-wise partition of the value table over the ranks of a
torch.distributed group (the paper's App. D).

Rank q holds rows [q R, min((q + 1) R, N)) of the physical table, R =
ceil(N / P).  Keys and queries are replicated, so each rank selects its own
tokens' slots (S1-S6).  The lookup then takes four steps:

  1. route:  the slots' shuffled rows (Eq. 14) grouped by owner (library kernel);
  2. all-to-all of the per-owner counts, then of the requested local rows;
  3. lookup: every rank reads the rows requested from its shard (library kernel);
  4. all-to-all of the rows back, then pool: the weighted sum of Eq. 15 over
     each slot's returned row and the IVE projection (library kernels).

Per rank and call the exchanges move 4 S (P - 1) / P bytes of indices and
S D_v es (P - 1) / P bytes of rows (S = n H m slots, es the storage bytes), the
paper's number-wise volumes with heads.  The local steps are an object with
``route(idx, P, R)``, ``lookup(rows)`` and ``pool(idx, w, slot_pos, rows)``;
``LibrarySteps`` runs them in the CUDA library.  This module holds only the
exchange and its bookkeeping.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


class LibrarySteps:
    """The local steps of one rank on a layer created over its shard
    (``cfg["shard_rows"]`` = the rows it holds)."""

    def __init__(self, layer):
        self.layer = layer

    def route(self, idx, P, rows_per_rank):
        return self.layer.shard_route(idx, P, rows_per_rank)

    def lookup(self, rows):
        return self.layer.shard_lookup(rows)

    def pool(self, idx, w, slot_pos, rows):
        return self.layer.shard_pool(idx, w, slot_pos, rows)


def rows_per_rank(n_rows: int, world: int) -> int:
    return (int(n_rows) + int(world) - 1) // int(world)


def shard_bounds(n_rows: int, world: int, rank: int):
    """First and one-past-last physical row rank `rank` holds."""
    R = rows_per_rank(n_rows, world)
    return min(rank * R, n_rows), min((rank + 1) * R, n_rows)


class NumberWiseTable:
    """The lookup-reduce (S7-S9) of one rank's slots against the table
    partitioned number-wise over `group`."""

    def __init__(self, steps, n_rows: int, d_v: int, group=None):
        self.steps = steps
        self.group = group
        self.P = dist.get_world_size(group)
        self.rank = dist.get_rank(group)
        self.R = rows_per_rank(n_rows, self.P)
        self.d_v = int(d_v)
        self.last = {}

    def lookup_reduce(self, idx: torch.Tensor, w: torch.Tensor) -> torch.Tensor:
        """out [n, D'_v] for this rank's slots idx [n, H, m] and weights w."""
        g = self.group
        counts, send_rows, slot_pos = self.steps.route(idx, self.P, self.R)
        send_counts = counts.to(torch.int64)
        recv_counts = torch.empty_like(send_counts)
        dist.all_to_all_single(recv_counts, send_counts, group=g)
        sc, rc = send_counts.tolist(), recv_counts.tolist()
        recv_rows = send_rows.new_empty(sum(rc))
        dist.all_to_all_single(recv_rows, send_rows, rc, sc, group=g)
        rows = self.steps.lookup(recv_rows)
        back = rows.new_empty((sum(sc), self.d_v))
        dist.all_to_all_single(back, rows, sc, rc, group=g)
        es = rows.element_size()
        self.last = {"slots": int(send_rows.numel()),
                     "index_bytes_sent": 4 * (sum(sc) - sc[self.rank]),
                     "row_bytes_sent": es * self.d_v * (sum(rc) - rc[self.rank]),
                     "requests_served": int(sum(rc))}
        return self.steps.pool(idx, w, slot_pos, back)
