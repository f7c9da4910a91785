"""Stochastic reduce and consensus error (oracle; test infrastructure only).

Paper passages followed:
* Eq. A.1, second line: each node replaces its model by the equal-weight
  average of its in-neighbours' half-step models, itself included.
* Section 3 ("stochastic reduce"): the reduce runs over a sparse graph
  instead of all nodes; written as W <- P W over the stacked models, with
  P = diag(d_in)^-1 A (Appendix A) or explicit doubly-stochastic weights.
* Appendix A, spectral-gap bound: ||P^t x - (1/n) 1|| <= sigma_2(P)^t; the
  consensus error ||W - 1 wbar^T||_F measures the distance to agreement.
"""
from __future__ import annotations

import numpy as np


def stochastic_reduce(H, nbr, wgt):
    """W[i] = sum_m wgt[i, m] * H[nbr[i, m]], summed in ascending-neighbour
    order, fp64; one output row per row of nbr."""
    H = np.asarray(H, dtype=np.float64)
    W = np.zeros((nbr.shape[0], H.shape[1]))
    for i in range(nbr.shape[0]):
        for m in range(nbr.shape[1]):
            W[i] += float(wgt[i, m]) * H[int(nbr[i, m])]
    return W


def reduce_with_matrix(H, P):
    """The same reduce written as one product W = P H with the dense N x N
    mixing matrix P (Appendix A); a library matmul serves as the step, so
    the fp64 summation order is the library's."""
    return np.asarray(P, dtype=np.float64) @ np.asarray(H, dtype=np.float64)


def consensus_error(W) -> float:
    """||W - 1 wbar^T||_F with wbar the mean over workers (rows)."""
    W = np.asarray(W, dtype=np.float64)
    wbar = W.mean(axis=0)
    return float(np.sqrt(((W - wbar) ** 2).sum()))
