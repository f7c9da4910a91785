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


# Relative distance from a bf16 midpoint within which the kernel's fp32
# residual may round either way.  The kernel forms R in fp32 from
# fp32-accumulated logits (errors of a few fp32 ulp, ~1e-6 relative at the
# bench shapes); 2^-16 (1.5e-5) covers that with a wide margin while
# flagging only ~1 % of the entries (a bf16 ulp is 2^-8 relative).
BF16_TIE_REL = 2.0 ** -16


def bf16_neighbours(R):
    """For fp64 values R: (nearest bf16 of fp32(R) as fp64, the other bf16
    neighbour of fp32(R) as fp64, |R - midpoint| / |R|)."""
    r32 = np.asarray(R, dtype=np.float32)
    u = r32.view(np.uint32).astype(np.uint64)
    lo = (u & np.uint64(0xFFFF0000)).astype(np.uint32)           # toward zero
    hi = (lo.astype(np.uint64) + np.uint64(0x10000)).astype(np.uint32)   # away from zero
    mid = (lo.astype(np.uint64) + np.uint64(0x8000)).astype(np.uint32)
    near = sgd.rne_bf16(r32)
    lo_f = lo.view(np.float32).astype(np.float64)
    hi_f = hi.view(np.float32).astype(np.float64)
    near_f = near.astype(np.float64)
    other = np.where(near_f == lo_f, hi_f, lo_f)
    dist = np.abs(np.asarray(R, np.float64) - mid.view(np.float32).astype(np.float64))
    return near_f, other, dist / np.maximum(np.abs(np.asarray(R, np.float64)), 1e-300)


def softmax_half_step_matching(Wm, H_gpu, Xbits, y, t, B, lr, l2, tol, tie_rel=BF16_TIE_REL):
    """Normwise relative error of one worker's half-step H_gpu [C, d] against
    the oracle (Eq. A.1 first line, bf16 rounding points mirrored), accepting
    either bf16 rounding of every residual entry whose fp64 value lies within
    tie_rel of a bf16 midpoint (the fp32 kernel and the fp64 oracle may
    round it differently, and identical classes move together).  Per class
    row, the flips that explain the difference are found by least squares
    over the flagged entries and rounded to {0, 1}.  Returns (error, oracle
    loss, number of flips used)."""
    X, R, loss = sgd.softmax_residual(Wm, Xbits, y, t, B)
    near, other, rel = bf16_neighbours(R)
    W64 = np.asarray(Wm, np.float64)
    H = W64 - lr * (near.T @ X + l2 * W64)
    H_gpu = np.asarray(H_gpu, np.float64)
    scale = max(np.abs(H).max(), 1e-30)
    D = H_gpu - H
    flips = 0
    if np.abs(D).max() > tol * scale:
        amb = rel <= tie_rel
        for c in np.nonzero(np.abs(D).max(axis=1) > 0.1 * tol * scale)[0]:
            bs = np.nonzero(amb[:, c])[0]
            if bs.shape[0] == 0:
                continue
            M = -lr * (other[bs, c] - near[bs, c])[:, None] * X[bs]     # one row per candidate flip
            s, *_ = np.linalg.lstsq(M.T, D[c], rcond=None)
            s = (s > 0.5).astype(np.float64)
            D[c] = D[c] - s @ M
            flips += int(s.sum())
    return float(np.abs(D).max() / scale), loss, flips
