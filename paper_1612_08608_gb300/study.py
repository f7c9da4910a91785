"""Graph comparison on one GB300: rounds, time and bytes to a target loss.

Section 6.1 compares ASAP's stochastic reduce over sparse graphs with the
all-reduce: sparse graphs need about as many iterations, while each worker
receives only its k in-neighbours' models per round instead of all N-1.
Here every graph runs the same workers, shards and model settings.  The
target is the loss the complete graph (the all-reduce) reaches after
``ref_rounds``, smoothed over one pass of the shards (``nb`` rounds).  For
each graph the study reports:

* the rounds to reach that target;
* the wall time per round on this GPU;
* the spectral gap 1 - sigma_2(P) of its mixing matrix (Section 3);
* the bytes each worker receives per round, k * d * 4 (the network cost the
  paper sets against the all-reduce's (N-1) * d * 4).

Run ``python -m paper_1612_08608_gb300.study`` (RCV1-shaped hinge SVM).
"""
from __future__ import annotations

import argparse
import json
import time

import numpy as np

from . import inputs
from .api import Context

# (name, graph kind, k, regenerated every round)
GRAPHS = (
    ("complete", "complete", None, False),
    ("root", "root", 2, False),
    ("ring", "ring", 1, False),
    ("random_regular_k2", "random_regular", 2, False),
    ("random_regular_k4_regen", "random_regular", 4, True),
)


def spectral_gap(nbr: np.ndarray, wgt: np.ndarray) -> float:
    """1 - sigma_2 of the mixing matrix P (row i: weights of its in-neighbours)."""
    N = nbr.shape[0]
    P = np.zeros((N, N))
    for i in range(N):
        for m in range(nbr.shape[1]):
            P[i, nbr[i, m]] += wgt[i, m]
    s = np.linalg.svd(P, compute_uv=False)
    return float(1.0 - s[1]) if N > 1 else 1.0


def _smoothed(losses: np.ndarray, window: int) -> np.ndarray:
    c = np.cumsum(np.concatenate([[0.0], losses.astype(np.float64)]))
    out = np.full(losses.shape[0], np.inf)
    out[window - 1:] = (c[window:] - c[:-window]) / window
    return out


def _context(shards, name, kind, k, regen, loss, B, lr, graph_seed):
    N = shards.N
    kk = N - 1 if k is None else k
    ctx = Context(N, shards.d, graph_seed=graph_seed, k=kk)
    ctx.set_model(loss, batch=B, lr=lr)
    ctx.set_graph(kind, regenerate=regen)
    ctx.load_shards(shards)
    return ctx, kk


def compare(shards, loss="hinge", B=256, lr=0.5, ref_rounds=400, max_rounds=4000, chunk=50, graph_seed=0,
            graphs=GRAPHS):
    """Returns one dict per graph (see the module docstring)."""
    nb = min(int(shards.rowptr[i].shape[0] - 1) // B for i in range(shards.N))
    window = max(1, nb)
    results = []
    target = None
    for name, kind, k, regen in graphs:
        ctx, kk = _context(shards, name, kind, k, regen, loss, B, lr, graph_seed)
        nbr, wgt = ctx.get_graph(0)
        limit = ref_rounds if target is None else max_rounds
        done, hit, t_run = 0, None, 0.0
        losses = np.empty(0, dtype=np.float32)
        while done < limit:
            n = min(chunk, limit - done)
            ctx.sync()
            t0 = time.perf_counter()
            ctx.round(n)
            ctx.sync()
            t_run += time.perf_counter() - t0
            lg, _ = ctx.read_metrics(done, n)
            losses = np.concatenate([losses, lg])
            done += n
            if target is not None:
                sm = _smoothed(losses, window)
                below = np.nonzero(sm <= target)[0]
                if below.shape[0]:
                    hit = int(below[0]) + 1
                    break
        if target is None:                      # the complete graph sets the target
            target = float(_smoothed(losses, window)[-1])
            hit = ref_rounds
        ctx.close()
        per_round_bytes = kk * shards.d * 4
        results.append({
            "graph": name, "k": kk, "spectral_gap": spectral_gap(nbr, wgt),
            "rounds_to_target": hit, "target_loss": target,
            "ms_per_round": 1e3 * t_run / max(done, 1),
            "bytes_per_worker_round": per_round_bytes,
            "bytes_per_worker_to_target": None if hit is None else per_round_bytes * hit,
        })
    return results


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workers", type=int, default=16)
    ap.add_argument("--rows", type=int, default=20000)
    ap.add_argument("--batch", type=int, default=256)
    ap.add_argument("--lr", type=float, default=0.5)
    ap.add_argument("--ref-rounds", type=int, default=400)
    ap.add_argument("--max-rounds", type=int, default=4000)
    args = ap.parse_args()
    sh = inputs.sparse_hinge_svm(seed=0, N=args.workers, rows=args.rows)
    res = compare(sh, "hinge", args.batch, args.lr, args.ref_rounds, args.max_rounds)
    for r in res:
        print(json.dumps(r))
    base = res[0]
    print("%-24s %3s %8s %10s %10s %14s" % ("graph", "k", "gap", "rounds", "ms/round", "bytes/worker"))
    for r in res:
        print("%-24s %3d %8.4f %10s %10.4f %14s" % (
            r["graph"], r["k"], r["spectral_gap"], r["rounds_to_target"], r["ms_per_round"],
            r["bytes_per_worker_to_target"]))
    print("target: smoothed loss %.5f (complete graph after %d rounds); all-reduce bytes per worker to target: %s"
          % (base["target_loss"], args.ref_rounds, base["bytes_per_worker_to_target"]))


if __name__ == "__main__":
    main()
