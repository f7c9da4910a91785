"""Host logic of the worker-sharded mode (Section 5, Implementation: one
process per group of workers, neighbour models sent point to point), on the
CPU: the partition, the exchange plan against a brute-force restatement and
closed forms, and whole runs of gloo ranks whose contexts are the oracle
(tests/sharded_fake.py), compared round by round with the unsharded oracle;
and failure detection made on the host: a rank that dies or hangs mid-run
ends its peer's round with an error instead of a wait without end."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

from oracle import graphs, rounds
from paper_1612_08608_gb300 import inputs
from paper_1612_08608_gb300.sharded import bytes_per_round, exchange_plan, owner_of, worker_ranges

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("N,world", [(8, 1), (8, 2), (7, 3), (64, 8), (5, 5)])
def test_worker_ranges_partition(N, world):
    r = worker_ranges(N, world)
    assert len(r) == world
    assert r[0][0] == 0 and sum(c for _, c in r) == N
    for (f0, c0), (f1, _) in zip(r, r[1:]):
        assert f1 == f0 + c0
    assert max(c for _, c in r) - min(c for _, c in r) <= 1
    own = owner_of(r, N)
    assert own.min() == 0 and own.max() == world - 1


def test_worker_ranges_reject_bad_world():
    with pytest.raises(ValueError):
        worker_ranges(4, 5)
    with pytest.raises(ValueError):
        worker_ranges(4, 0)


def _brute_plan(nbr, ranges, rank):
    """Messages as (sender, receiver, row) triples by direct enumeration of
    every table entry: worker i on rank a lists j on rank b != a."""
    N = nbr.shape[0]
    own = [next(r for r, (f, c) in enumerate(ranges) if f <= i < f + c) for i in range(N)]
    msgs = set()
    for i in range(N):
        for j in nbr[i]:
            if own[int(j)] != own[i]:
                msgs.add((own[int(j)], own[i], int(j)))
    send = {q: sorted(j for s, t, j in msgs if s == rank and t == q) for q in range(len(ranges))}
    recv = {q: sorted(j for s, t, j in msgs if s == q and t == rank) for q in range(len(ranges))}
    return {q: v for q, v in send.items() if v}, {q: v for q, v in recv.items() if v}


@pytest.mark.parametrize("kind,N,k,world", [("random_regular", 16, 4, 3), ("root", 16, 2, 4),
                                             ("complete", 6, 5, 2), ("ring", 9, 1, 4), ("identity", 5, 0, 2)])
def test_exchange_plan_matches_brute_force(kind, N, k, world):
    ranges = worker_ranges(N, world)
    for rnd in range(3):
        nbr, _ = graphs.build_graph(kind, N, k, 7, rnd)
        for rank in range(world):
            send, recv = exchange_plan(nbr, ranges, rank)
            bs, br = _brute_plan(nbr, ranges, rank)
            assert {q: list(v) for q, v in send.items()} == bs
            assert {q: list(v) for q, v in recv.items()} == br
            # what rank sends to q is what q expects from rank
            for q in range(world):
                if q != rank:
                    got = exchange_plan(nbr, ranges, q)[1].get(rank, np.zeros(0, np.int32))
                    assert list(send.get(q, [])) == list(got)


def test_exchange_closed_forms():
    N, d = 64, 1000
    for world in (2, 4, 8):
        ranges = worker_ranges(N, world)
        # directed ring (i <- i-1): each range's first worker needs the
        # previous range's last, so every rank sends one row per round
        assert bytes_per_round(graphs.ring_graph(N), ranges, d) == [4 * d] * world
        # complete graph: every rank sends all of its rows to every other rank
        full = graphs.complete_graph(N)
        assert bytes_per_round(full, ranges, d) == [4 * d * c * (world - 1) for _, c in ranges]
    # identity graph: nothing to send
    assert bytes_per_round(graphs.identity_graph(8), worker_ranges(8, 4), d) == [0, 0, 0, 0]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, cfg, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch.distributed as dist
    from sharded_fake import OracleShardContext
    from paper_1612_08608_gb300 import inputs as inp
    from paper_1612_08608_gb300.sharded import ShardedWorkers
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        sh = inp.sparse_hinge_svm(seed=cfg["seed"], N=cfg["N"], d=cfg["d"], rows=cfg["rows"], mean_nnz=20.0)
        ctx = OracleShardContext(sh, cfg["B"], cfg["loss"], cfg["lr"], cfg["k"], cfg["kind"], cfg["graph_seed"],
                                 cfg["regen"])
        run = ShardedWorkers(ctx, rank, world)
        run.setup()
        per_round = []
        for _ in range(cfg["T"]):
            run.round()
            per_round.append(ctx.W[run.first:run.first + run.count].copy())
        out.put((rank, run.first, per_round, run.sent_bytes))
    finally:
        dist.barrier()
        dist.destroy_process_group()


@pytest.mark.parametrize("world,kind,k,regen", [(2, "random_regular", 2, True), (3, "root", 2, False),
                                                (2, "ring", 1, False)])
def test_sharded_ranks_match_unsharded_oracle_gloo(world, kind, k, regen):
    cfg = dict(seed=3, N=6, d=400, rows=128, B=32, loss="hinge", lr=0.5, k=k, kind=kind, graph_seed=5,
               regen=regen, T=6)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, cfg, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=300) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    sh = inputs.sparse_hinge_svm(seed=cfg["seed"], N=cfg["N"], d=cfg["d"], rows=cfg["rows"], mean_nnz=20.0)
    sched = rounds.graph_schedule(kind, cfg["N"], k, cfg["graph_seed"], regen)
    W = np.zeros((cfg["N"], cfg["d"]))
    sent = 0
    for t in range(cfg["T"]):
        nbr, wgt = sched(t)
        W, _, _ = rounds.sparse_round(W, sh, t, cfg["B"], cfg["loss"], cfg["lr"], nbr, wgt)
        for rank, first, per_round, _ in res:
            got = per_round[t]
            assert np.array_equal(got, W[first:first + got.shape[0]]), (t, rank)
        sent += sum(bytes_per_round(nbr, worker_ranges(cfg["N"], world), cfg["d"])) * 2   # fp64 rows
    assert sum(r[3] for r in res) == sent


def _failing_rank_main(rank, world, port, cfg, fail_rank, fail_round, out, mode="raise"):
    """A rank whose local step fails at round `fail_round`: mode "raise"
    leaves at once, without tearing down the group (a crashed process);
    mode "stall" reports, then stays alive without sending anything for
    longer than the group's timeout (a hung process)."""
    import datetime
    import time
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch.distributed as dist
    from sharded_fake import OracleShardContext
    from paper_1612_08608_gb300 import inputs as inp
    from paper_1612_08608_gb300.sharded import ShardedWorkers
    t0 = time.monotonic()
    err, t = None, -1
    try:
        dist.init_process_group("gloo", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=cfg.get("pg_timeout_s", 20)))
        sh = inp.sparse_hinge_svm(seed=cfg["seed"], N=cfg["N"], d=cfg["d"], rows=cfg["rows"], mean_nnz=20.0)
        ctx = OracleShardContext(sh, cfg["B"], cfg["loss"], cfg["lr"], cfg["k"], cfg["kind"], cfg["graph_seed"],
                                 cfg["regen"])
        if rank == fail_rank:
            step = ctx.local_step

            def local_step():
                if ctx.t == fail_round:
                    if mode == "stall":
                        out.put((rank, "stalled", time.monotonic() - t0, ctx.t))
                        out.close()
                        out.join_thread()
                        time.sleep(2 * cfg.get("pg_timeout_s", 20) + 1)
                        os._exit(3)
                    raise RuntimeError("injected failure")
                step()
            ctx.local_step = local_step
        run = ShardedWorkers(ctx, rank, world)
        run.setup()
        try:
            for _ in range(cfg["T"]):
                run.round()
        except Exception as e:             # the failure itself, or a peer's lost message
            err = type(e).__name__
        t = run.t
    except Exception as e:                 # set-up failed: report it, do not leave the parent waiting
        err = "setup " + repr(e)
    out.put((rank, err, time.monotonic() - t0, t))
    out.close()
    out.join_thread()                      # flushed before the process ends
    os._exit(3 if rank == fail_rank else 0)


@pytest.mark.parametrize("mode", ["raise", "stall"])
def test_a_failed_rank_ends_its_peers_round_with_an_error_gloo(mode):
    # rank 1 fails at the start of round 2, before sending its rows: it
    # dies ("raise": rank 0's receive sees the connection close) or hangs
    # ("stall": the group's 4 s timeout ends rank 0's receive); either way
    # rank 0 gets an error instead of waiting forever, at the same round
    cfg = dict(seed=3, N=6, d=400, rows=128, B=32, loss="hinge", lr=0.5, k=1, kind="ring", graph_seed=5,
               regen=False, T=6, pg_timeout_s=4)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_failing_rank_main, args=(r, 2, port, cfg, 1, 2, q, mode)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        res = sorted(q.get(timeout=180) for _ in procs)
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():
                p.kill()
    (r0, err0, dt0, t0), (r1, err1, dt1, t1) = res
    assert (r0, r1) == (0, 1)
    assert err1 == ("stalled" if mode == "stall" else "RuntimeError") and t1 == 2
    assert err0 is not None and not err0.startswith("setup") and t0 == 2, (err0, t0)
    assert dt0 < 60
    if mode == "stall":      # the error came from the timeout, after the stall began
        assert dt0 >= dt1 + 2, (dt0, dt1)
    assert procs[0].exitcode == 0 and procs[1].exitcode == 3
