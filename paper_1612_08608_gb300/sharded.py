"""Worker-sharded ASAP across processes (Section 5, Implementation).

Each process steps a contiguous range of the N workers in its own context
(``Context.set_worker_range``).  In every round a worker's half-step model
x_j - eta g_j goes, as a point-to-point message, to each process that owns
one of its out-neighbours under the round's graph; the receiver's reduce may
run once every in-neighbour of its workers has arrived (the host-side form
of NOTIFY).  Every process builds the same graph from the shared seed, so
both ends of a message agree on its rows without any control traffic.

The messages travel as host buffers through ``torch.distributed``
point-to-point calls (gloo here; any backend with CPU send/recv).  All
arithmetic of the round stays in the context's kernels: this module only
plans and moves rows.
"""
from __future__ import annotations

from typing import Dict, List, Sequence, Tuple

import numpy as np


def worker_ranges(N: int, world: int) -> List[Tuple[int, int]]:
    """Contiguous (first, count) per rank; counts differ by at most one."""
    if world < 1 or world > N:
        raise ValueError("need 1 <= world <= N")
    base, extra = divmod(N, world)
    out, first = [], 0
    for r in range(world):
        c = base + (1 if r < extra else 0)
        out.append((first, c))
        first += c
    return out


def owner_of(ranges: Sequence[Tuple[int, int]], N: int) -> np.ndarray:
    own = np.full(N, -1, dtype=np.int64)
    for r, (f, c) in enumerate(ranges):
        own[f:f + c] = r
    if (own < 0).any():
        raise ValueError("ranges do not cover [0, N)")
    return own


def exchange_plan(nbr: np.ndarray, ranges: Sequence[Tuple[int, int]], rank: int):
    """Rows this rank sends to / receives from each peer in one round.

    nbr is the round's [N, k+1] in-neighbour table (row i lists the workers
    whose models worker i averages).  send[q] = the owned workers that some
    worker of rank q lists; recv[q] = the workers of rank q that some owned
    worker lists.  Both sorted, so that sender and receiver agree on order.
    """
    nbr = np.asarray(nbr, dtype=np.int64)
    N = nbr.shape[0]
    own = owner_of(ranges, N)
    send: Dict[int, np.ndarray] = {}
    recv: Dict[int, np.ndarray] = {}
    for q in range(len(ranges)):
        if q == rank:
            continue
        fq, cq = ranges[q]
        fr, cr = ranges[rank]
        want_by_q = np.unique(nbr[fq:fq + cq].ravel())
        s = want_by_q[own[want_by_q] == rank]
        want_by_me = np.unique(nbr[fr:fr + cr].ravel())
        v = want_by_me[own[want_by_me] == q]
        if s.size:
            send[q] = s.astype(np.int32)
        if v.size:
            recv[q] = v.astype(np.int32)
    return send, recv


def bytes_per_round(nbr: np.ndarray, ranges: Sequence[Tuple[int, int]], P: int) -> List[int]:
    """Bytes each rank sends in one round (fp32 rows of P parameters)."""
    return [4 * P * sum(int(v.size) for v in exchange_plan(nbr, ranges, r)[0].values())
            for r in range(len(ranges))]


class ShardedWorkers:
    """One rank of a worker-sharded run over a context that steps this
    rank's range of workers.

    ``ctx`` needs: N, P, row_dtype, set_worker_range, local_step, read_rows,
    write_rows, stochastic_reduce, get_graph (a ``Context`` of this package).  Call
    ``setup`` before the context's shards are loaded, then ``round`` once per
    round on every rank.
    """

    def __init__(self, ctx, rank: int, world: int, group=None, first_round: int = 0):
        self.ctx, self.rank, self.world, self.group = ctx, rank, world, group
        self.ranges = worker_ranges(ctx.N, world)
        self.first, self.count = self.ranges[rank]
        self.t = first_round
        self.sent_bytes = 0
        self.recv_bytes = 0

    def setup(self):
        self.ctx.set_worker_range(self.first, self.count)

    def owned(self) -> range:
        return range(self.first, self.first + self.count)

    def shard_list(self, full):
        """A per-worker list with None outside this rank's range (for load_shards)."""
        return [a if self.first <= i < self.first + self.count else None for i, a in enumerate(full)]

    def round(self):
        import torch
        import torch.distributed as dist
        ctx = self.ctx
        nbr, _ = ctx.get_graph(self.t)
        send, recv = exchange_plan(nbr, self.ranges, self.rank)
        ctx.local_step()
        # The rows go as stored: both ends keep the same lazy L2 scale (every
        # context applies the same schedule), so the scale is not sent.
        reqs, inbox, outbox = [], {}, []
        for q in sorted(recv):
            buf = torch.from_numpy(np.empty((recv[q].size, ctx.P), dtype=ctx.row_dtype))
            inbox[q] = buf
            reqs.append(dist.irecv(buf, src=q, group=self.group))
        for q in sorted(send):
            rows, _ = ctx.read_rows(send[q])
            outbox.append(torch.from_numpy(rows))   # alive until every request is done
            reqs.append(dist.isend(outbox[-1], dst=q, group=self.group))
            self.sent_bytes += rows.nbytes
        for rq in reqs:
            rq.wait()
        if inbox:
            rows = np.concatenate([recv[q] for q in sorted(inbox)])
            vals = np.concatenate([inbox[q].numpy() for q in sorted(inbox)])
            ctx.write_rows(rows, vals)
            self.recv_bytes += vals.nbytes
        ctx.stochastic_reduce()
        self.t += 1
