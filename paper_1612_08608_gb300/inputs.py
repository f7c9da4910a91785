"""Seeded synthetic inputs shaped like the paper's workloads.

This module only *draws data*: feature matrices, labels, initial parameters.
It holds none of the method's arithmetic (no margins, losses, gradients,
mixing or graph construction), so the CPU oracle and the CUDA path can both
be fed from it without sharing any of the computation they are compared on.

The paper trains linear SVMs on RCV1, webspam and splice-site and a CNN on
CIFAR-10 (Section 6, "Evaluation").  None of those datasets is available here;
the generators below stand in for them with the same shapes, sparsity
patterns and value distributions:

* ``tiny_dense_logistic``   -- d=64 dense N(0,1) rows stored as CSR.
* ``sparse_hinge_svm``      -- RCV1-like: d=47,236, lognormal row lengths
  (mean 75, clipped to [5, 1000]), Zipf(1.1) column popularity, tf-idf-like
  positive values, L2-normalised rows.
* ``sparse_logistic_hashed``-- hashed features: d=2^20, 100 distinct uniform
  column ids per row, N(0,1) values.
* ``mixing_params``         -- W ~ N(0,1) for the stochastic-reduce sweep.
* ``dense_softmax``         -- d=2048 bf16 N(0,1) features, C classes from the
  argmax of x.W*^T plus Gumbel noise.

All randomness is numpy PCG64 keyed by (seed, purpose, worker) so that any
worker's shard can be regenerated on its own.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

__all__ = [
    "SparseShards", "DenseShards", "WORKLOADS",
    "tiny_dense_logistic", "sparse_hinge_svm", "sparse_logistic_hashed",
    "sparse_custom", "mixing_params", "mixing_params_device", "dense_softmax", "bf16_bits_to_f32",
]

# Stream ids keep the draws for different purposes independent.
_TEACHER, _ROWLEN, _COLS, _VALS, _FLIPS, _PARAMS, _GUMBEL, _X = range(8)


def _rng(seed: int, purpose: int, worker: int = -1) -> np.random.Generator:
    return np.random.default_rng([int(seed), int(purpose), int(worker) + 1])


@dataclass
class SparseShards:
    """Per-worker CSR shards.  Row r of worker i spans
    ``col[i][rowptr[i][r]:rowptr[i][r+1]]``; labels are +1/-1 float32."""
    d: int
    rowptr: List[np.ndarray] = field(default_factory=list)  # int64 [rows+1]
    col: List[np.ndarray] = field(default_factory=list)     # int32 [nnz]
    val: List[np.ndarray] = field(default_factory=list)     # float32 [nnz]
    y: List[np.ndarray] = field(default_factory=list)       # float32 [rows]

    @property
    def N(self) -> int:
        return len(self.rowptr)

    def n_rows(self, i: int) -> int:
        return int(self.rowptr[i].shape[0] - 1)

    def nnz(self, i: int) -> int:
        return int(self.rowptr[i][-1])


@dataclass
class DenseShards:
    """Per-worker dense shards: X as raw bf16 bits [rows, d] (uint16), labels
    as class ids in [0, C)."""
    d: int
    C: int
    X: List[np.ndarray] = field(default_factory=list)  # uint16 [rows, d]
    y: List[np.ndarray] = field(default_factory=list)  # int32 [rows]

    @property
    def N(self) -> int:
        return len(self.X)

    def n_rows(self, i: int) -> int:
        return int(self.X[i].shape[0])


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32 (a bit shift)."""
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    # Input conversion only: the features are *defined* as bf16 values, so
    # the library cast decides them (round-to-nearest-even).
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()


def _labels_from_teacher(scores: np.ndarray, flip: float, rng: np.random.Generator) -> np.ndarray:
    y = np.where(scores >= 0.0, 1.0, -1.0).astype(np.float32)   # sign(0) -> +1
    flips = rng.random(y.shape[0]) < flip
    y[flips] = -y[flips]
    return y


def _row_scores(rowptr: np.ndarray, col: np.ndarray, val: np.ndarray, wstar: np.ndarray) -> np.ndarray:
    n = rowptr.shape[0] - 1
    row_of = np.repeat(np.arange(n), np.diff(rowptr))
    return np.bincount(row_of, weights=val.astype(np.float64) * wstar[col], minlength=n)


def _per_worker(fn, N):
    """fn(i) for every worker, on a thread pool (each worker has its own
    streams, so the result does not depend on the pool)."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(max_workers=max(1, min(N, os.cpu_count() or 1, 16))) as ex:
        return list(ex.map(fn, range(N)))


def _distinct_columns(rng: np.random.Generator, lengths: np.ndarray, sample) -> tuple:
    """Draw ``lengths[r]`` distinct column ids for every row r with ``sample(m)``
    (which returns m iid ids); duplicates inside a row are redrawn until none
    remain.  Returns (rowptr, col) with each row's ids sorted ascending."""
    n = lengths.shape[0]
    rowptr = np.zeros(n + 1, dtype=np.int64)
    np.cumsum(lengths, out=rowptr[1:])
    row_of = np.repeat(np.arange(n, dtype=np.int64), lengths)
    col = sample(row_of.shape[0]).astype(np.int64)
    pos = np.arange(row_of.shape[0])            # entries still under inspection
    while pos.shape[0]:
        order = np.lexsort((col[pos], row_of[pos]))
        p_s = pos[order]
        r_s, c_s = row_of[p_s], col[p_s]
        dup = np.zeros(p_s.shape[0], dtype=bool)
        dup[1:] = (r_s[1:] == r_s[:-1]) & (c_s[1:] == c_s[:-1])
        if not dup.any():
            break
        col[p_s[dup]] = sample(int(dup.sum())).astype(np.int64)
        bad_rows = np.unique(r_s[dup])
        pos = p_s[np.isin(r_s, bad_rows)]       # only rows that had a duplicate
    order = np.lexsort((col, row_of))
    return rowptr, col[order].astype(np.int32)


# ---------------------------------------------------------------------------
# Workload 1: tiny dense logistic regression (N=4 ring, d=64, 256 rows/worker)
# ---------------------------------------------------------------------------
def tiny_dense_logistic(seed: int = 0, N: int = 4, d: int = 64, rows: int = 256,
                        flip: float = 0.05) -> SparseShards:
    """Dense N(0,1) features stored as CSR with every column present."""
    wstar = _rng(seed, _TEACHER).standard_normal(d)
    out = SparseShards(d=d)
    for i in range(N):
        x = _rng(seed, _VALS, i).standard_normal((rows, d)).astype(np.float32)
        rowptr = np.arange(0, rows * d + 1, d, dtype=np.int64)
        col = np.tile(np.arange(d, dtype=np.int32), rows)
        val = x.reshape(-1)
        scores = x.astype(np.float64) @ wstar
        out.rowptr.append(rowptr)
        out.col.append(col)
        out.val.append(val)
        out.y.append(_labels_from_teacher(scores, flip, _rng(seed, _FLIPS, i)))
    return out


# ---------------------------------------------------------------------------
# Workload 2: RCV1-shaped sparse hinge SVM
# ---------------------------------------------------------------------------
def sparse_hinge_svm(seed: int = 0, N: int = 16, d: int = 47236, rows: int = 20000,
                     mean_nnz: float = 75.0, sigma: float = 1.0, lo: int = 5, hi: int = 1000,
                     zipf_a: float = 1.1, flip: float = 0.03, label_skew: float = 0.0) -> SparseShards:
    """Lognormal row lengths with the given mean, Zipf(a) column popularity
    over ranks 1..d (column id = rank-1), tf-idf-like values
    ``Exp(1) * ln(1 + d/(col+1))``, rows scaled to unit L2 norm.

    ``label_skew`` in [0, 1) makes the shards heterogeneous by label: worker
    i keeps a share 1/2 + label_skew (i/(N-1) - 1/2) of positive rows (drawn
    from a pool of twice the rows), so that workers see different class
    balances, as data split by source would."""
    ranks = np.arange(1, d + 1, dtype=np.float64)
    cdf = np.cumsum(ranks ** (-zipf_a))
    cdf /= cdf[-1]
    wstar = _rng(seed, _TEACHER).standard_normal(d)
    mu = np.log(mean_nnz) - 0.5 * sigma * sigma
    out = SparseShards(d=d)

    pool = rows if label_skew == 0.0 else 2 * rows

    def one(i):
        sh_i = _hinge_pool(i)
        if label_skew == 0.0:
            return sh_i
        rowptr, col, val, y = sh_i
        frac = 0.5 + label_skew * ((i / (N - 1) if N > 1 else 0.5) - 0.5)
        pos, neg = np.nonzero(y > 0)[0], np.nonzero(y < 0)[0]
        n_pos = min(int(round(frac * rows)), pos.shape[0])
        n_neg = rows - n_pos
        if n_neg > neg.shape[0]:
            n_neg = neg.shape[0]
            n_pos = rows - n_neg
        srng = _rng(seed, _FLIPS + 100, i)
        keep = np.concatenate([srng.choice(pos, n_pos, replace=False), srng.choice(neg, n_neg, replace=False)])
        keep = keep[srng.permutation(keep.shape[0])]
        lens = np.diff(rowptr)[keep]
        rp = np.zeros(rows + 1, dtype=np.int64)
        np.cumsum(lens, out=rp[1:])
        idx = np.concatenate([np.arange(rowptr[r], rowptr[r + 1]) for r in keep]) if rows else np.zeros(0, np.int64)
        return rp, col[idx], val[idx], y[keep]

    def _hinge_pool(i):
        lengths = np.rint(_rng(seed, _ROWLEN, i).lognormal(mu, sigma, pool)).astype(np.int64)
        lengths = np.clip(lengths, lo, min(hi, d))
        crng = _rng(seed, _COLS, i)

        def sample(m, crng=crng):
            return np.minimum(np.searchsorted(cdf, crng.random(m), side="right"), d - 1)

        rowptr, col = _distinct_columns(crng, lengths, sample)
        raw = _rng(seed, _VALS, i).exponential(1.0, col.shape[0]) * np.log1p(d / (col.astype(np.float64) + 1.0))
        row_of = np.repeat(np.arange(pool), lengths)
        norms = np.sqrt(np.bincount(row_of, weights=raw * raw, minlength=pool))
        val = (raw / norms[row_of]).astype(np.float32)
        return rowptr, col, val, _labels_from_teacher(_row_scores(rowptr, col, val, wstar), flip,
                                                      _rng(seed, _FLIPS, i))

    for rowptr, col, val, y in _per_worker(one, N):
        out.rowptr.append(rowptr)
        out.col.append(col)
        out.val.append(val)
        out.y.append(y)
    return out


# ---------------------------------------------------------------------------
# Workload 3: hashed sparse logistic regression at scale
# ---------------------------------------------------------------------------
def sparse_logistic_hashed(seed: int = 0, N: int = 64, d: int = 1 << 20, rows: int = 50000,
                           nnz: int = 100, flip: float = 0.03) -> SparseShards:
    """Exactly ``nnz`` distinct uniform column ids per row, N(0,1) values."""
    wstar = _rng(seed, _TEACHER).standard_normal(d)
    out = SparseShards(d=d)

    def one(i):
        crng = _rng(seed, _COLS, i)
        col = crng.integers(0, d, size=(rows, nnz), dtype=np.int32)
        col.sort(axis=1)
        while True:
            bad = np.nonzero((np.diff(col, axis=1) == 0).any(axis=1))[0]
            if bad.shape[0] == 0:
                break
            col[bad] = crng.integers(0, d, size=(bad.shape[0], nnz), dtype=np.int32)
            col[bad] = np.sort(col[bad], axis=1)
        col = col.reshape(-1)
        val = _rng(seed, _VALS, i).standard_normal(rows * nnz, dtype=np.float32)
        rowptr = np.arange(0, rows * nnz + 1, nnz, dtype=np.int64)
        scores = (val.astype(np.float64) * wstar[col]).reshape(rows, nnz).sum(axis=1)
        return rowptr, col, val, _labels_from_teacher(scores, flip, _rng(seed, _FLIPS, i))

    for rowptr, col, val, y in _per_worker(one, N):
        out.rowptr.append(rowptr)
        out.col.append(col)
        out.val.append(val)
        out.y.append(y)
    return out


def sparse_custom(seed: int, N: int, d: int, rows: int, lengths: Optional[list] = None,
                  max_len: int = 40, hot_col: Optional[int] = None, flip: float = 0.05,
                  positive: bool = False) -> SparseShards:
    """Small ragged shards for edge cases: per-row lengths drawn uniformly
    from [0, max_len] (empty rows included) unless ``lengths`` (one array per
    worker) is given; ``hot_col`` forces one column into every non-empty row."""
    wstar = _rng(seed, _TEACHER).standard_normal(d)
    out = SparseShards(d=d)
    for i in range(N):
        if lengths is not None:
            ln = np.asarray(lengths[i], dtype=np.int64)
        else:
            ln = _rng(seed, _ROWLEN, i).integers(0, max_len + 1, rows).astype(np.int64)
        ln = np.minimum(ln, d)
        crng = _rng(seed, _COLS, i)
        rowptr, col = _distinct_columns(crng, ln, lambda m, crng=crng: crng.integers(0, d, m))
        if hot_col is not None:
            # Replace each non-empty row's first id by hot_col unless present.
            for r in range(ln.shape[0]):
                a, b = rowptr[r], rowptr[r + 1]
                if b > a and hot_col not in col[a:b]:
                    col[a] = hot_col
                    col[a:b] = np.sort(col[a:b])
        v = _rng(seed, _VALS, i).standard_normal(col.shape[0]).astype(np.float32)
        if positive:
            v = np.abs(v)
        out.rowptr.append(rowptr)
        out.col.append(col.astype(np.int32))
        out.val.append(v)
        out.y.append(_labels_from_teacher(_row_scores(rowptr, col, v, wstar), flip, _rng(seed, _FLIPS, i)))
    return out


# ---------------------------------------------------------------------------
# Workload 4: parameters for the stochastic-reduce sweep
# ---------------------------------------------------------------------------
def mixing_params(seed: int, N: int, d: int, rows: Optional[range] = None,
                  cols: Optional[np.ndarray] = None) -> np.ndarray:
    """W ~ N(0,1) float32 [N, d], one independent stream per worker row.
    ``rows``/``cols`` select a sub-block without materialising the rest of a
    row only when ``cols`` is None; with ``cols`` the full row is drawn and
    then indexed (the stream defines the row)."""
    rr = range(N) if rows is None else rows
    ncol = d if cols is None else cols.shape[0]
    W = np.empty((len(rr), ncol), dtype=np.float32)
    for a, i in enumerate(rr):
        row = _rng(seed, _PARAMS, i).standard_normal(d, dtype=np.float32)
        W[a] = row if cols is None else row[cols]
    return W


def mixing_params_device(seed: int, N: int, d: int, device="cuda"):
    """W ~ N(0,1) float32 [N, d] drawn on a CUDA device with torch's seeded
    generator (Philox), for sweep sizes whose host draw would take minutes
    (up to 256 x 10^7 values).  A different stream from ``mixing_params``;
    a sub-block for the oracle is read back from the returned tensor."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) * 1000003 + 7919)
    return torch.randn((N, d), generator=g, device=device, dtype=torch.float32)


# ---------------------------------------------------------------------------
# Workload 5: dense softmax regression with bf16 features
# ---------------------------------------------------------------------------
def dense_softmax(seed: int = 0, N: int = 32, d: int = 2048, C: int = 1000,
                  rows: int = 25600) -> DenseShards:
    """x ~ N(0,1) rounded to bf16; W* ~ N(0, 1/d) [C, d]; label =
    argmax_c(x.W*_c + Gumbel(0,1)) (ties to the lowest id)."""
    import torch
    Wstar = (_rng(seed, _TEACHER).standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    Wt = torch.from_numpy(Wstar)
    out = DenseShards(d=d, C=C)
    for i in range(N):
        xf = _rng(seed, _X, i).standard_normal((rows, d), dtype=np.float32)
        bits = _f32_to_bf16_bits(xf)
        xs = torch.from_numpy(bf16_bits_to_f32(bits))
        scores = (xs @ Wt.T).numpy().astype(np.float64)
        scores += _rng(seed, _GUMBEL, i).gumbel(0.0, 1.0, scores.shape)
        out.X.append(bits)
        out.y.append(np.argmax(scores, axis=1).astype(np.int32))
    return out


# Named workloads with the sizes the paper's experiments are shaped like.
WORKLOADS = {
    "tiny_dense_logistic": dict(N=4, d=64, rows=256, B=32, loss="logistic", lr=0.1, rounds=10,
                                graph="explicit_ring_half_quarter", k=2),
    "sparse_hinge_svm": dict(N=16, d=47236, rows=20000, B=256, loss="hinge", lr=0.1, rounds=50,
                             graph="random_regular", k=2, regenerate=False),
    "sparse_logistic_hashed": dict(N=64, d=1 << 20, rows=50000, B=512, loss="logistic", lr=0.1,
                                   rounds=100, graph="random_regular", k=4, regenerate=True),
    "mixing_sweep": dict(N=(8, 32, 128, 256), d=(100000, 1000000, 10000000), k=(1, 2, 4, "N-1"),
                         rounds=20),
    "dense_softmax": dict(N=32, d=2048, C=1000, rows=25600, B=512, loss="softmax", lr=0.1,
                          rounds=50, graph="root", k=2),
}
