"""GPU parity of the worker-sharded mode (Section 5, Implementation): contexts
that each step a range of the workers and exchange half-step rows, against
the unsharded oracle round by round (1e-5 normwise per worker), through the
C ABI.  Two ways of running the ranks: two contexts in one process (rows
moved by the test), and two processes on the one GPU with gloo moving the
rows (paper_1612_08608_gb300.sharded).  The kernels of one context never
wait on another context's flags: a worker stepped elsewhere is announced by
the host, when its row is written."""
import datetime
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

from oracle import rounds
from paper_1612_08608_gb300 import inputs
from paper_1612_08608_gb300.sharded import exchange_plan, worker_ranges
from parity import sparse_round_matching

pytestmark = pytest.mark.gpu

TOL = 1e-5
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _shards(cfg):
    return inputs.sparse_hinge_svm(seed=cfg["seed"], N=cfg["N"], d=cfg["d"], rows=cfg["rows"], mean_nnz=30.0)


def _make(cfg, sh, first, count):
    from paper_1612_08608_gb300 import Context
    ctx = Context(cfg["N"], cfg["d"], graph_seed=cfg["graph_seed"], k=cfg["k"])
    ctx.set_model(cfg["loss"], batch=cfg["B"], lr=cfg["lr"], l2=cfg.get("l2", 0.0))
    ctx.set_schedule(cfg.get("tau", 1))
    ctx.set_graph(cfg["kind"], regenerate=cfg["regen"])
    ctx.set_shard_residency(cfg.get("residency", "device"))
    if count != cfg["N"]:
        ctx.set_worker_range(first, count)
    keep = lambda arrs: [a if first <= i < first + count else None for i, a in enumerate(arrs)]
    ctx.load_shards(rowptr=keep(sh.rowptr), col=keep(sh.col), val=keep(sh.val), y=keep(sh.y))
    return ctx


def _owned_rows(ctx, first, count):
    rows, scale = ctx.read_rows(np.arange(first, first + count))
    assert scale == 1.0      # between rounds the rows hold true values
    return rows


CASES = [
    dict(seed=3, N=6, d=1000, rows=256, B=32, loss="hinge", lr=0.5, k=2, kind="random_regular", graph_seed=5,
         regen=True, T=8),
    dict(seed=4, N=7, d=777, rows=320, B=40, loss="logistic", lr=0.3, k=2, kind="root", graph_seed=1,
         regen=False, T=6, tau=2, l2=1e-3, residency="host"),
    dict(seed=5, N=6, d=512, rows=192, B=32, loss="logistic", lr=0.3, k=5, kind="complete", graph_seed=0,
         regen=False, T=4),
]


@pytest.mark.parametrize("cfg", CASES, ids=["hinge-regen", "logistic-tau2-l2-host", "complete"])
def test_two_contexts_in_one_process_match_oracle(cfg):
    sh = _shards(cfg)
    N, world = cfg["N"], 2
    ranges = worker_ranges(N, world)
    ctxs = [_make(cfg, sh, f, c) for f, c in ranges]
    tau, l2 = cfg.get("tau", 1), cfg.get("l2", 0.0)
    W_t = np.zeros((N, cfg["d"]))
    for t in range(cfg["T"]):
        nbr, wgt = ctxs[0].get_graph(t)
        for c in ctxs:
            c.local_step()
        for r, c in enumerate(ctxs):
            send, _ = exchange_plan(nbr, ranges, r)
            for q, rows in send.items():
                vals, scale = c.read_rows(rows)
                assert scale == pytest.approx(np.prod([1 - cfg["lr"] * l2] * tau), rel=1e-6)
                ctxs[q].write_rows(rows, vals)
        for c in ctxs:
            c.stochastic_reduce()
        W_n = np.concatenate([_owned_rows(c, f, n) for c, (f, n) in zip(ctxs, ranges)])
        err, lref, _ = sparse_round_matching(W_t, W_n, sh, t, cfg["B"], cfg["loss"], cfg["lr"],
                                             nbr.astype(np.int64), wgt.astype(np.float64), TOL, l2=l2, tau=tau)
        assert err <= TOL, (t, err)
        shares = [c.read_metrics(t, 1) for c in ctxs]
        assert abs(sum(s[0][0] for s in shares) - lref) <= 1e-5 * max(1.0, abs(lref)), t
        assert all(np.isnan(s[1][0]) for s in shares)
        W_t = W_n.astype(np.float64)
    for c, (_, n) in zip(ctxs, ranges):
        cnt = c.read_counters()
        assert cnt["reduces"] == n * cfg["T"] and cnt["timeouts"] == 0


def test_reduce_refuses_a_missing_row_then_recovers():
    cfg = CASES[0]
    sh = _shards(cfg)
    ranges = worker_ranges(cfg["N"], 2)
    ctxs = [_make(cfg, sh, f, c) for f, c in ranges]
    from paper_1612_08608_gb300.api import AsapError
    nbr, wgt = ctxs[0].get_graph(0)
    for c in ctxs:
        c.local_step()
    with pytest.raises(AsapError) as e:
        ctxs[0].stochastic_reduce()
    assert e.value.name == "ASAP_ERR_ARG"
    with pytest.raises(AsapError):                  # an owned row is not deliverable
        ctxs[0].write_rows([0], np.zeros((1, cfg["d"]), np.float32))
    for r, c in enumerate(ctxs):
        for q, rows in exchange_plan(nbr, ranges, r)[0].items():
            ctxs[q].write_rows(rows, c.read_rows(rows)[0])
    for c in ctxs:
        c.stochastic_reduce()
    W_n = np.concatenate([_owned_rows(c, f, n) for c, (f, n) in zip(ctxs, ranges)])
    err, _, _ = sparse_round_matching(np.zeros((cfg["N"], cfg["d"])), W_n, sh, 0, cfg["B"], cfg["loss"], cfg["lr"],
                                      nbr.astype(np.int64), wgt.astype(np.float64), TOL)
    assert err <= TOL
    assert ctxs[0].read_counters()["timeouts"] == 0


def test_whole_range_is_the_unsharded_context():
    cfg = CASES[0]
    sh = _shards(cfg)
    a = _make(cfg, sh, 0, cfg["N"])
    b = _make(cfg, sh, 0, cfg["N"])
    b.set_worker_range(0, cfg["N"])            # drops the shards: load again
    b.load_shards(sh)
    a.round(3)
    b.round(3)
    assert np.array_equal(a.read_params()[0], b.read_params()[0])


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, cfg, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    from paper_1612_08608_gb300 import Context, inputs as inp
    from paper_1612_08608_gb300.sharded import ShardedWorkers
    # a rank that fails ends the other's pending receive within two minutes
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=120))
    try:
        sh = inp.sparse_hinge_svm(seed=cfg["seed"], N=cfg["N"], d=cfg["d"], rows=cfg["rows"], mean_nnz=30.0)
        ctx = Context(cfg["N"], cfg["d"], graph_seed=cfg["graph_seed"], k=cfg["k"])
        ctx.set_model(cfg["loss"], batch=cfg["B"], lr=cfg["lr"])
        ctx.set_graph(cfg["kind"], regenerate=cfg["regen"])
        run = ShardedWorkers(ctx, rank, world)
        run.setup()
        ctx.load_shards(rowptr=run.shard_list(sh.rowptr), col=run.shard_list(sh.col), val=run.shard_list(sh.val),
                        y=run.shard_list(sh.y))
        per_round = []
        for _ in range(cfg["T"]):
            run.round()
            per_round.append(ctx.read_rows(np.arange(run.first, run.first + run.count))[0])
        out.put((rank, run.first, per_round, None))
    except Exception as e:                        # report, do not hang the parent
        out.put((rank, -1, None, repr(e)))
    finally:
        dist.destroy_process_group()


def test_two_processes_gloo_share_the_gpu():
    cfg = dict(seed=6, N=8, d=2000, rows=320, B=64, loss="hinge", lr=0.5, k=2, kind="random_regular",
               graph_seed=2, regen=True, T=10)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, cfg, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=600) for _ in procs]
    for p in procs:
        p.join(timeout=120)
    assert all(r[3] is None for r in res), [r[3] for r in res]
    assert all(p.exitcode == 0 for p in procs)
    res.sort(key=lambda r: r[0])
    sh = _shards(cfg)
    sched = rounds.graph_schedule(cfg["kind"], cfg["N"], cfg["k"], cfg["graph_seed"], cfg["regen"])
    W_t = np.zeros((cfg["N"], cfg["d"]))
    for t in range(cfg["T"]):
        nbr, wgt = sched(t)
        W_n = np.concatenate([r[2][t] for r in res])
        err, _, _ = sparse_round_matching(W_t, W_n, sh, t, cfg["B"], cfg["loss"], cfg["lr"], nbr, wgt, TOL)
        assert err <= TOL, (t, err)
        W_t = W_n.astype(np.float64)
