"""The tie-aware check of the dense half-step (tests/parity.py), on the CPU:
a half-step in which the residual entries near a bf16 midpoint are rounded
the other way -- as an fp32 kernel may do -- is accepted, and a half-step with
one entry rounded the wrong way far from a midpoint, or with a dropped L2
term, is rejected.  The mistakes are planted in the oracle's own arithmetic."""
import numpy as np

from oracle import rounds, sgd
from paper_1612_08608_gb300 import inputs
from parity import BF16_TIE_REL, bf16_neighbours, softmax_half_step_matching


def _tied_case():
    # From W = 0, every class absent from the first minibatch gets the same
    # row of W_1; in the next minibatch their residuals are exactly equal.
    N, d, C, B, lr = 1, 64, 40, 16, 0.5
    sh = inputs.dense_softmax(seed=3, N=N, d=d, C=C, rows=2 * B)
    nbr, wgt = np.zeros((1, 1), np.int64), np.ones((1, 1))
    W1, _, _ = rounds.softmax_round(np.zeros((N, C * d), np.float32), sh, 0, B, lr, nbr, wgt)
    return sh, W1.astype(np.float32)[0].reshape(C, d), B, lr


def _half_step(Wm, X, R, lr, l2):
    W64 = Wm.astype(np.float64)
    return W64 - lr * (R.T @ X + l2 * W64)


def test_flipped_near_ties_are_accepted():
    sh, Wm, B, lr = _tied_case()
    X, R, _ = sgd.softmax_residual(Wm, sh.X[0], sh.y[0], 1, B)
    near, other, rel = bf16_neighbours(R)
    # widen the band for the test so that several entries are flagged
    amb = rel <= BF16_TIE_REL * 64
    assert amb.sum() > 0
    R_alt = np.where(amb, other, near)
    H_alt = _half_step(Wm, X, R_alt, lr, 0.0)
    err, _, flips = softmax_half_step_matching(Wm, H_alt, sh.X[0], sh.y[0], 1, B, lr, 0.0, 1e-6,
                                               tie_rel=BF16_TIE_REL * 64)
    assert err <= 1e-6 and flips == int(amb.sum())


def test_wrong_rounding_far_from_a_tie_is_rejected():
    sh, Wm, B, lr = _tied_case()
    X, R, _ = sgd.softmax_residual(Wm, sh.X[0], sh.y[0], 1, B)
    near, other, rel = bf16_neighbours(R)
    b, c = np.unravel_index(np.argmax(rel), rel.shape)         # the entry farthest from a midpoint
    R_bad = near.copy()
    R_bad[b, c] = other[b, c]
    H_bad = _half_step(Wm, X, R_bad, lr, 0.0)
    err, _, _ = softmax_half_step_matching(Wm, H_bad, sh.X[0], sh.y[0], 1, B, lr, 0.0, 1e-6)
    assert err > 1e-6
    H_nol2 = _half_step(Wm, X, near, lr, 0.0)
    err, _, _ = softmax_half_step_matching(Wm, H_nol2, sh.X[0], sh.y[0], 1, B, lr, 0.05, 1e-6)
    assert err > 1e-6
    err, _, flips = softmax_half_step_matching(Wm, _half_step(Wm, X, near, lr, 0.05), sh.X[0], sh.y[0], 1, B, lr,
                                               0.05, 1e-12)
    assert err <= 1e-12 and flips == 0
