"""Comparison helpers shared by the GPU parity tests."""
import itertools

import numpy as np

from oracle import rounds, sgd


def rel_err_rows(W_gpu, W_ref):
    """max over workers of ||w_gpu - w_ref||_inf / ||w_ref||_inf."""
    W_gpu = np.asarray(W_gpu, dtype=np.float64)
    W_ref = np.asarray(W_ref, dtype=np.float64)
    num = np.abs(W_gpu - W_ref).max(axis=1)
    den = np.maximum(np.abs(W_ref).max(axis=1), 1e-30)
    return float((num / den).max())


def hinge_near_ties(W, shards, t, B, tol=1e-5):
    """{worker: [rows]} whose y*m is within tol of the hinge corner at W."""
    out = {}
    for i in range(shards.N):
        b0, _ = sgd.batch_window(t, shards.n_rows(i), B)
        m = sgd.sparse_margins(shards.rowptr[i], shards.col[i], shards.val[i], W[i], b0, B)
        z = shards.y[i][b0:b0 + B] * m
        rows = list(np.nonzero(np.abs(1.0 - z) < tol)[0])
        if rows:
            out[i] = rows
    return out


def sparse_round_matching(W_t, W_gpu_next, shards, t, B, loss, lr, nbr, wgt, tol, l2=0.0, tau=1, lr_at=None):
    """Oracle round from the GPU's W_t; on hinge corner rows accept either
    subgradient (one local step per round only).  Returns (rel_err, oracle
    loss, oracle consensus)."""
    ties = hinge_near_ties(W_t, shards, t, B) if (loss == "hinge" and tau == 1) else {}
    cands = [{}]
    if ties:
        flat = [(i, r) for i, rows in ties.items() for r in rows]
        assert len(flat) <= 6, "too many hinge corner rows to enumerate"
        cands = []
        for mask in itertools.product([0, 1], repeat=len(flat)):
            f = {}
            for (i, r), on in zip(flat, mask):
                if on:
                    f.setdefault(i, []).append(r)
            cands.append(f)
    best = None
    for flips in cands:
        Wn, lval, cons = rounds.sparse_round(W_t, shards, t, B, loss, lr, nbr, wgt, l2=l2, flips=flips, tau=tau,
                                             lr_at=lr_at)
        e = rel_err_rows(W_gpu_next, Wn)
        if best is None or e < best[0]:
            best = (e, lval, cons)
        if e <= tol:
            break
    return best
