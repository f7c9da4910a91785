"""One local minibatch SGD step per worker (oracle; test infrastructure only).

Paper passages followed:
* Eq. A.1, first line: w_{t+1/2} = w_t - eta_t * grad f_i(w_t).
* Section 5 (Implementation): each replica trains its own model on a
  handful of local examples between two exchanges.
* Section 6 (Evaluation): the linear SVM of Bottou's SVM-SGD (hinge loss).

Readings where the paper is silent (stated in the design notes):
* minibatch of round t = rows [(t mod nb) B, (t mod nb) B + B) of the
  worker's shard, nb = floor(rows / B) (sequential windows, tail dropped);
* grad f_i = (1/B) sum_b r_b x_b + l2 * w, r_b = d loss / d margin;
* hinge: loss = max(0, 1 - y m); r = -y if y m < 1 else 0 (strict);
* logistic: loss = ln(1 + exp(-y m)); r = -y * sigmoid(-y m);
* softmax regression (dense bf16 variant): loss = logsumexp(z) - z_y,
  R = (softmax(z) - e_y) / B, with the bf16 rounding points of the tensor-core
  path mirrored: W is read as RNE_bf16(W), R is formed in fp32 and rounded to
  bf16 before the gradient product; everything else is fp64.

All arithmetic is fp64 on fp32 (or bf16) inputs.
"""
from __future__ import annotations

import numpy as np


def batch_window(t: int, n_rows: int, B: int):
    """First and one-past-last row of round t's minibatch."""
    nb = n_rows // B
    if nb <= 0:
        raise ValueError("shard has fewer rows than one minibatch")
    b0 = (t % nb) * B
    return b0, b0 + B


def _batch_rows(rowptr, b0, B):
    lens = np.diff(rowptr[b0:b0 + B + 1]).astype(np.int64)
    return np.repeat(np.arange(B), lens), int(rowptr[b0]), int(rowptr[b0 + B])


def sparse_margins(rowptr, col, val, w, b0, B):
    """m_b = x_b . w for the B rows starting at b0."""
    row_of, lo, hi = _batch_rows(rowptr, b0, B)
    prod = val[lo:hi].astype(np.float64) * np.asarray(w, dtype=np.float64)[col[lo:hi]]
    return np.bincount(row_of, weights=prod, minlength=B)


def loss_and_derivative(loss: str, y, m, flip_rows=()):
    """Per-row loss and r_b = d loss / d m_b.  ``flip_rows`` inverts the hinge
    branch on the listed rows (used only to accept either subgradient on rows
    whose y*m is within rounding of the hinge corner)."""
    y = np.asarray(y, dtype=np.float64)
    z = y * m
    if loss == "hinge":
        active = z < 1.0
        for b in flip_rows:
            active[b] = not active[b]
        lval = np.maximum(0.0, 1.0 - z)
        r = np.where(active, -y, 0.0)
    elif loss == "logistic":
        lval = np.logaddexp(0.0, -z)
        r = -y / (1.0 + np.exp(z))            # -y * sigmoid(-z)
    else:
        raise ValueError("unknown loss %r" % loss)
    return lval, r


def sparse_gradient(rowptr, col, val, r, b0, B, d):
    """(1/B) sum_b r_b x_b as a dense length-d vector."""
    row_of, lo, hi = _batch_rows(rowptr, b0, B)
    return np.bincount(col[lo:hi], weights=r[row_of] * val[lo:hi].astype(np.float64), minlength=d) / B


def learning_rate(kind: str, eta0: float, gamma: float, k: int) -> float:
    """eta_k of local step k (Eq. A.1 writes the rate as eta_t): ``constant``
    keeps eta0; ``inverse`` is eta0 / (1 + gamma k), the decreasing rate of
    Bottou's SVM-SGD, which the paper's SVM experiments use (Section 6)."""
    if kind == "constant":
        return float(eta0)
    if kind == "inverse":
        return float(eta0) / (1.0 + float(gamma) * k)
    raise ValueError("unknown learning-rate schedule %r" % kind)


def local_step(w, g, lr, l2=0.0):
    """Eq. A.1 first line, with an optional L2 term in f_i."""
    w = np.asarray(w, dtype=np.float64)
    return w - lr * (g + l2 * w)


def sparse_worker_step(w, rowptr, col, val, y, t, B, loss, lr, l2=0.0, flip_rows=()):
    """Returns (w_{t+1/2}, mean minibatch loss at w_t, r) for one worker."""
    d = w.shape[0]
    b0, _ = batch_window(t, rowptr.shape[0] - 1, B)
    m = sparse_margins(rowptr, col, val, w, b0, B)
    lval, r = loss_and_derivative(loss, y[b0:b0 + B], m, flip_rows)
    g = sparse_gradient(rowptr, col, val, r, b0, B, d)
    return local_step(w, g, lr, l2), float(lval.mean()), m


# ---------------------------------------------------------------------------
# bf16 helpers and the dense softmax-regression step
# ---------------------------------------------------------------------------
def rne_bf16(x) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even), returned as
    float32.  bf16 keeps the top 16 bits of the float32 encoding; the
    discarded low half decides the rounding.  Finite inputs only."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep_lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + keep_lsb) & np.uint64(0xFFFF0000)
    return u.astype(np.uint32).view(np.float32)


def bf16_to_f64(bits) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def softmax_residual(Wm, Xbits, y, t, B, mirror_bf16=True):
    """The minibatch of round t for one worker: returns (X_b fp64 [B, d],
    R = (softmax(X_b Wread^T) - onehot(y_b)) / B fp64 [B, C] before any
    rounding, mean loss at W_t).  Wread = RNE_bf16(Wm) when mirroring the
    tensor-core path, else Wm."""
    b0, _ = batch_window(t, Xbits.shape[0], B)
    X = bf16_to_f64(Xbits[b0:b0 + B])
    yb = np.asarray(y[b0:b0 + B], dtype=np.int64)
    Wread = rne_bf16(Wm).astype(np.float64) if mirror_bf16 else np.asarray(Wm, dtype=np.float64)
    Z = X @ Wread.T                                   # [B, C] logits
    zmax = Z.max(axis=1, keepdims=True)
    E = np.exp(Z - zmax)
    S = E.sum(axis=1, keepdims=True)
    lse = zmax[:, 0] + np.log(S[:, 0])
    loss = lse - Z[np.arange(B), yb]
    Pm = E / S
    Pm[np.arange(B), yb] -= 1.0
    return X, Pm / B, float(loss.mean())


def softmax_worker_step(Wm, Xbits, y, t, B, lr, mirror_bf16=True, l2=0.0):
    """Dense softmax regression for one worker.  Wm: [C, d] float32 master
    weights; Xbits: [rows, d] bf16 bits; y: [rows] class ids.  Returns
    (W_{t+1/2} fp64 [C, d], mean loss at W_t)."""
    X, R, loss = softmax_residual(Wm, Xbits, y, t, B, mirror_bf16)
    if mirror_bf16:
        R = rne_bf16(R.astype(np.float32)).astype(np.float64)
    G = R.T @ X                                       # [C, d]
    H = np.asarray(Wm, dtype=np.float64) - lr * (G + l2 * np.asarray(Wm, dtype=np.float64))
    return H, loss
