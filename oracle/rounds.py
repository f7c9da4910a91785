"""Whole ASAP rounds (oracle; test infrastructure only).

Eq. A.1 applied once per round t, in the paper's order: every worker i takes
its SGD step on its own shard, then every worker averages the half-step
models of its in-neighbours (W <- P_t W).  W_0 = 0 unless given (Appendix A
takes w_0 = 0).  Per round the oracle records the mean over workers of the
minibatch loss at the pre-step model and the consensus error after the reduce.

``graph`` is a callable rnd -> (nbr, wgt) so that a graph regenerated every
round (Section 3.1: such graphs are cheap to build afresh) and a fixed one
look the same here.
"""
from __future__ import annotations

import numpy as np

from . import graphs, reduce, sgd


def graph_schedule(kind: str, N: int, k: int, graph_seed: int = 0, regenerate: bool = False,
                   explicit=None):
    """rnd -> (nbr, wgt).  ``explicit`` = (nbr, wgt) arrays for a user graph."""
    if kind == "explicit":
        nbr, wgt = explicit
        nbr = np.asarray(nbr, dtype=np.int64)
        wgt = np.asarray(wgt, dtype=np.float64)
        return lambda rnd: (nbr, wgt)
    fixed = None if regenerate else graphs.build_graph(kind, N, k, graph_seed, 0)
    if fixed is not None:
        return lambda rnd: fixed
    return lambda rnd: graphs.build_graph(kind, N, k, graph_seed, rnd)


def sparse_round(W, shards, t, B, loss, lr, nbr, wgt, l2=0.0, flips=None, tau=1, lr_at=None):
    """One round from W_t (any float array [N, d]); returns
    (W_{t+1} fp64, mean minibatch loss, consensus error of W_{t+1}).

    Each worker takes ``tau`` local steps before the reduce (Section 5: the
    replicas exchange models after a handful of local examples): step j of round t
    is global step k = t*tau + j, on minibatch k and at rate lr_at(k) (``lr``
    when lr_at is None).  The loss is the workers' mean minibatch loss of the
    round's last step, at its pre-step model.  ``flips`` maps a worker to the
    hinge rows of its last step whose subgradient branch is inverted."""
    N = W.shape[0]
    H = np.empty(W.shape, dtype=np.float64)
    losses = []
    for i in range(N):
        h = np.asarray(W[i], dtype=np.float64)
        for j in range(tau):
            k = t * tau + j
            eta = lr if lr_at is None else lr_at(k)
            fl = (flips or {}).get(i, ()) if j == tau - 1 else ()
            h, lval, _ = sgd.sparse_worker_step(h, shards.rowptr[i], shards.col[i], shards.val[i],
                                                shards.y[i], k, B, loss, eta, l2, fl)
        H[i] = h
        losses.append(lval)
    Wn = reduce.stochastic_reduce(H, nbr, wgt)
    return Wn, float(np.mean(losses)), reduce.consensus_error(Wn)


def run_sparse(shards, T, B, loss, lr, graph, W0=None, l2=0.0, t0=0, tau=1, lr_at=None):
    """Free-running trajectory: returns (W_T fp64, losses[T], consensus[T])."""
    N, d = shards.N, shards.d
    W = np.zeros((N, d)) if W0 is None else np.asarray(W0, dtype=np.float64)
    losses, cons = [], []
    for t in range(t0, t0 + T):
        nbr, wgt = graph(t)
        W, lval, c = sparse_round(W, shards, t, B, loss, lr, nbr, wgt, l2, tau=tau, lr_at=lr_at)
        losses.append(lval)
        cons.append(c)
    return W, np.array(losses), np.array(cons)


def softmax_round(W, shards, t, B, lr, nbr, wgt, l2=0.0, mirror_bf16=True):
    """W: float32 master weights [N, C*d] (row i = worker i's C x d matrix,
    class-major).  Returns (W_{t+1} fp64, mean loss, consensus error)."""
    N = W.shape[0]
    C, d = shards.C, shards.d
    H = np.empty(W.shape, dtype=np.float64)
    losses = []
    for i in range(N):
        Wm = np.asarray(W[i], dtype=np.float32).reshape(C, d)
        h, lval = sgd.softmax_worker_step(Wm, shards.X[i], shards.y[i], t, B, lr, mirror_bf16, l2)
        H[i] = h.reshape(-1)
        losses.append(lval)
    Wn = reduce.stochastic_reduce(H, nbr, wgt)
    return Wn, float(np.mean(losses)), reduce.consensus_error(Wn)


def run_softmax(shards, T, B, lr, graph, W0=None, l2=0.0, t0=0, lr_at=None):
    """Free-running dense trajectory from W0 (default 0); the master weights
    are fp32 between rounds, as on the tensor-core path.  Returns
    (W_T fp64, losses[T], consensus[T])."""
    N, P = shards.N, shards.C * shards.d
    W = np.zeros((N, P), np.float32) if W0 is None else np.asarray(W0, dtype=np.float32)
    losses, cons = [], []
    for t in range(t0, t0 + T):
        nbr, wgt = graph(t)
        eta = lr if lr_at is None else lr_at(t)
        Wn, lval, c = softmax_round(W, shards, t, B, eta, nbr, wgt, l2)
        W = Wn.astype(np.float32)
        losses.append(lval)
        cons.append(c)
    return Wn, np.array(losses), np.array(cons)


def mixing_rounds(W0, T, graph, t0=0):
    """Stochastic reduce alone, T times; returns (W_T fp64, consensus[T])."""
    W = np.asarray(W0, dtype=np.float64)
    cons = []
    for t in range(t0, t0 + T):
        nbr, wgt = graph(t)
        W = reduce.stochastic_reduce(W, nbr, wgt)
        cons.append(reduce.consensus_error(W))
    return W, np.array(cons)
