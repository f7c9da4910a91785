"""Pins for oracle/sgd.py and oracle/rounds.py (no GPU).

* A hand-computed hinge step, including the hinge corner y*m = 1 (strict <).
* Central finite differences of the minibatch loss for logistic, hinge (off
  the corner) and softmax regression: the gradient is the loss's derivative.
* First step from W_0 = 0 in closed form for all three losses.
* bf16 round-to-nearest-even against torch's float32 -> bfloat16 cast.
* N = 1 reduces to textbook minibatch SGD written with dense matrices.
* The complete graph reduces to all-reduce SGD on the concatenated batch
  (Section 3: stochastic reduce converges to the same result as all-reduce).
* Eq. A.2: with d = 1, w_0 = 0 and a fixed gradient sequence,
  w_t = -sum_k eta_k P^{t-k} g_k, which fixes the order "SGD, then reduce".
* The early-exit permutation sampler is uniform over admissible layers.
* Learning-rate schedules at literal values; two local steps per round by
  hand (inverse rate, with and without L2); one worker with tau local steps
  equals textbook minibatch SGD over the global step sequence.
* A hand-computed softmax step from a W that bf16 cannot represent: the
  logits read RNE_bf16(W), R is rounded to bf16, the fp32 master is updated.
* rounds.softmax_round against a restatement with dense matrices (step with
  torch's bf16 casts, then P H with P written out, the loss and consensus).
"""
import itertools
import math

import numpy as np
import pytest

from oracle import graphs, reduce, rounds, sgd
from paper_1612_08608_gb300 import inputs


def _csr(rows, d):
    rowptr = [0]
    col, val = [], []
    for r in rows:
        for c, v in sorted(r.items()):
            col.append(c)
            val.append(v)
        rowptr.append(len(col))
    return np.array(rowptr, np.int64), np.array(col, np.int32), np.array(val, np.float32)


def test_hand_computed_hinge_step():
    # w = [0.5, -1, 0, 2], eta = 0.3, B = 3
    # row 0: y=+1, x={0:1, 3:0.5}:      m = 1.5,  y m = 1.5  -> r = 0,  loss 0
    # row 1: y=+1, x={1:0.25, 2:1}:     m = -0.25, y m = -0.25 -> r = -1, loss 1.25
    # row 2: y=-1, x={0:1, 1:1, 3:-0.25}: m = -1, y m = 1 (corner, strict <) -> r = 0, loss 0
    # g = -(1/3) x_1 = [0, -1/12, -1/3, 0];  w - 0.3 g = [0.5, -0.975, 0.1, 2]
    rowptr, col, val = _csr([{0: 1.0, 3: 0.5}, {1: 0.25, 2: 1.0}, {0: 1.0, 1: 1.0, 3: -0.25}], 4)
    y = np.array([1, 1, -1], np.float32)
    w = np.array([0.5, -1.0, 0.0, 2.0])
    h, loss, m = sgd.sparse_worker_step(w, rowptr, col, val, y, 0, 3, "hinge", 0.3)
    assert np.array_equal(m, [1.5, -0.25, -1.0])
    assert h == pytest.approx([0.5, -0.975, 0.1, 2.0], abs=1e-15)
    assert loss == pytest.approx(1.25 / 3, abs=1e-15)
    # flipping the corner row's branch adds r = +1 times x_2 / 3
    h2, _, _ = sgd.sparse_worker_step(w, rowptr, col, val, y, 0, 3, "hinge", 0.3, flip_rows=(2,))
    assert h2 == pytest.approx([0.5 - 0.1, -0.975 - 0.1, 0.1, 2.0 + 0.025], abs=1e-15)


def test_hand_computed_logistic_step():
    rowptr, col, val = _csr([{0: 1.0, 3: 0.5}, {1: 0.25, 2: 1.0}, {0: 1.0, 1: 1.0, 3: -0.25}], 4)
    y = np.array([1, 1, -1], np.float32)
    w = np.array([0.5, -1.0, 0.0, 2.0])
    h, loss, _ = sgd.sparse_worker_step(w, rowptr, col, val, y, 0, 3, "logistic", 0.3)
    z = [1.5, -0.25, 1.0]                        # y * m per row
    r = [-yy / (1.0 + math.exp(zz)) for yy, zz in zip((1.0, 1.0, -1.0), z)]
    g = [(r[0] * 1.0 + r[2] * 1.0) / 3, (r[1] * 0.25 + r[2] * 1.0) / 3, r[1] / 3,
         (r[0] * 0.5 + r[2] * -0.25) / 3]
    assert h == pytest.approx([w[j] - 0.3 * g[j] for j in range(4)], abs=1e-15)
    assert loss == pytest.approx(sum(math.log1p(math.exp(-zz)) for zz in z) / 3, abs=1e-15)


def test_batch_window_wraps_and_drops_tail():
    assert sgd.batch_window(0, 100, 32) == (0, 32)
    assert sgd.batch_window(2, 100, 32) == (64, 96)
    assert sgd.batch_window(3, 100, 32) == (0, 32)      # nb = 3, the 4 tail rows are never used
    with pytest.raises(ValueError):
        sgd.batch_window(0, 10, 32)


def _mean_loss_sparse(w, sh, i, t, B, loss):
    b0, _ = sgd.batch_window(t, sh.n_rows(i), B)
    m = sgd.sparse_margins(sh.rowptr[i], sh.col[i], sh.val[i], w, b0, B)
    lval, _ = sgd.loss_and_derivative(loss, sh.y[i][b0:b0 + B], m)
    return lval.mean()


@pytest.mark.parametrize("loss", ["logistic", "hinge"])
def test_sparse_gradient_is_derivative_of_minibatch_loss(loss):
    sh = inputs.sparse_custom(seed=3, N=1, d=30, rows=40, max_len=8)
    rng = np.random.default_rng(0)
    w = rng.standard_normal(30) * 0.3
    lr, B, t = 0.5, 16, 1
    h, _, m = sgd.sparse_worker_step(w, sh.rowptr[0], sh.col[0], sh.val[0], sh.y[0], t, B, loss, lr)
    g = (w - h) / lr
    if loss == "hinge":
        b0, _ = sgd.batch_window(t, 40, B)
        assert np.min(np.abs(1 - sh.y[0][b0:b0 + B] * m)) > 1e-3   # off the corner
    eps = 1e-6
    for j in range(30):
        e = np.zeros(30)
        e[j] = eps
        fd = (_mean_loss_sparse(w + e, sh, 0, t, B, loss) - _mean_loss_sparse(w - e, sh, 0, t, B, loss)) / (2 * eps)
        assert g[j] == pytest.approx(fd, abs=1e-7)


def test_softmax_gradient_is_derivative_of_minibatch_loss():
    sh = inputs.dense_softmax(seed=1, N=1, d=12, C=5, rows=16)
    rng = np.random.default_rng(1)
    Wm = (rng.standard_normal((5, 12)) * 0.2).astype(np.float32)
    lr, B = 0.25, 8

    def L(Wd):
        X = sgd.bf16_to_f64(sh.X[0][:B])
        Z = X @ Wd.T
        zmax = Z.max(axis=1, keepdims=True)
        lse = zmax[:, 0] + np.log(np.exp(Z - zmax).sum(axis=1))
        return float((lse - Z[np.arange(B), sh.y[0][:B]]).mean())

    H, loss = sgd.softmax_worker_step(Wm, sh.X[0], sh.y[0], 0, B, lr, mirror_bf16=False)
    G = (Wm.astype(np.float64) - H) / lr
    assert loss == pytest.approx(L(Wm.astype(np.float64)), abs=1e-14)
    eps = 1e-6
    for (c, j) in [(0, 0), (1, 5), (4, 11), (2, 7), (3, 3)]:
        E = np.zeros((5, 12))
        E[c, j] = eps
        W0 = Wm.astype(np.float64)
        fd = (L(W0 + E) - L(W0 - E)) / (2 * eps)
        assert G[c, j] == pytest.approx(fd, abs=1e-8)


def test_first_step_from_zero_closed_forms():
    sh = inputs.sparse_custom(seed=5, N=1, d=20, rows=12, max_len=6)
    B, lr = 12, 0.1
    Xd = np.zeros((12, 20))
    for r in range(12):
        a, b = sh.rowptr[0][r], sh.rowptr[0][r + 1]
        Xd[r, sh.col[0][a:b]] = sh.val[0][a:b]
    yx = (sh.y[0][:, None].astype(np.float64) * Xd).sum(axis=0)
    h, loss, _ = sgd.sparse_worker_step(np.zeros(20), sh.rowptr[0], sh.col[0], sh.val[0], sh.y[0], 0, B, "hinge", lr)
    assert h == pytest.approx(lr / B * yx, abs=1e-15) and loss == 1.0
    h, loss, _ = sgd.sparse_worker_step(np.zeros(20), sh.rowptr[0], sh.col[0], sh.val[0], sh.y[0], 0, B, "logistic", lr)
    assert h == pytest.approx(lr / (2 * B) * yx, abs=1e-15) and loss == pytest.approx(math.log(2.0))
    dsh = inputs.dense_softmax(seed=2, N=1, d=6, C=4, rows=8)
    X = sgd.bf16_to_f64(dsh.X[0])
    E = np.zeros((8, 4))
    E[np.arange(8), dsh.y[0]] = 1.0
    want = -(lr / 8) * (np.full((8, 4), 0.25) - E).T @ X
    H, loss = sgd.softmax_worker_step(np.zeros((4, 6), np.float32), dsh.X[0], dsh.y[0], 0, 8, lr)
    assert H == pytest.approx(want, abs=1e-15)       # R = (1/4 - e_y)/8 is exact in bf16
    assert loss == pytest.approx(math.log(4.0))


def test_rne_bf16_matches_library_cast():
    import torch
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(100000).astype(np.float32),
        (rng.standard_normal(1000) * 1e-30).astype(np.float32),
        (rng.standard_normal(1000) * 1e30).astype(np.float32),
        # exact ties: bit 15 set, bits 0..14 clear, both parities of bit 16
        (np.arange(4096, dtype=np.uint32) << 16 | 0x8000).view(np.float32),
        np.array([0.0, -0.0, 1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8], np.float32),
    ])
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    got = sgd.rne_bf16(x)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def test_single_worker_is_textbook_minibatch_sgd():
    sh = inputs.sparse_custom(seed=7, N=1, d=25, rows=64, max_len=10)
    B, lr, T = 16, 0.2, 6
    sched = rounds.graph_schedule("identity", 1, 0)
    Wo, losses, _ = rounds.run_sparse(sh, T, B, "logistic", lr, sched)
    # dense restatement: w <- w - lr/B * X_b^T (-y * sigmoid(-y * X_b w))
    Xd = np.zeros((64, 25))
    for r in range(64):
        a, b = sh.rowptr[0][r], sh.rowptr[0][r + 1]
        Xd[r, sh.col[0][a:b]] = sh.val[0][a:b]
    y = sh.y[0].astype(np.float64)
    w = np.zeros(25)
    for t in range(T):
        b0 = (t % 4) * B
        Xb, yb = Xd[b0:b0 + B], y[b0:b0 + B]
        s = 1.0 / (1.0 + np.exp(yb * (Xb @ w)))
        w = w - lr / B * (Xb.T @ (-yb * s))
    assert Wo[0] == pytest.approx(w, abs=1e-14)


def test_complete_graph_equals_allreduce_sgd():
    N, B, lr, T = 4, 8, 0.3, 5
    sh = inputs.sparse_custom(seed=9, N=N, d=15, rows=32, max_len=7)
    Wo, _, cons = rounds.run_sparse(sh, T, B, "hinge", lr, rounds.graph_schedule("complete", N, N - 1))
    # one model, gradient averaged over all N workers' minibatches
    w = np.zeros(15)
    for t in range(T):
        gs = []
        for i in range(N):
            h, _, _ = sgd.sparse_worker_step(w, sh.rowptr[i], sh.col[i], sh.val[i], sh.y[i], t, B, "hinge", lr)
            gs.append((w - h) / lr)
        w = w - lr * np.mean(gs, axis=0)
    for i in range(N):
        assert Wo[i] == pytest.approx(w, abs=1e-13)
    assert np.all(cons < 1e-13)


def test_unrolled_form_eq_a2():
    N, T = 6, 7
    nbr, wgt = graphs.build_graph("random_regular", N, 2, graph_seed=11)
    P = graphs.mixing_matrix(nbr, wgt)
    rng = np.random.default_rng(3)
    g = rng.standard_normal((T, N))
    eta = 0.5 / (1.0 + np.arange(T))
    w = np.zeros((N, 1))
    for t in range(T):
        w = reduce.stochastic_reduce(sgd.local_step(w, g[t][:, None], eta[t]), nbr, wgt)
        want = -sum(eta[k] * np.linalg.matrix_power(P, t + 1 - k) @ g[k] for k in range(t + 1))
        assert w[:, 0] == pytest.approx(want, abs=1e-13)


def test_admissible_layer_sampler_is_uniform():
    # N = 4 after a fixed cycle 0->1->2->3->0: admissible sigma avoid i and i-1.
    in_nbrs = [{3}, {0}, {1}, {2}]
    admissible = [p for p in itertools.permutations(range(4))
                  if all(p[i] != i and p[i] not in in_nbrs[i] for i in range(4))]
    rng = graphs.SplitMix64(21)
    counts = {}
    accepted = 0
    while accepted < 20000:
        s = graphs._admissible_permutation(rng, in_nbrs)
        if s is not None:
            counts[tuple(s)] = counts.get(tuple(s), 0) + 1
            accepted += 1
    assert set(counts) == set(admissible)
    exp = accepted / len(admissible)
    chi2 = sum((c - exp) ** 2 / exp for c in counts.values())
    assert chi2 < 25.0


def test_learning_rate_schedules():
    assert [sgd.learning_rate("constant", 0.3, 7.0, k) for k in (0, 1, 50)] == [0.3, 0.3, 0.3]
    # eta0 / (1 + gamma k) with eta0 = 0.5, gamma = 0.25
    assert [sgd.learning_rate("inverse", 0.5, 0.25, k) for k in (0, 4, 12)] == [0.5, 0.25, 0.125]
    with pytest.raises(ValueError):
        sgd.learning_rate("step", 0.5, 0.1, 0)


def test_hand_computed_two_local_steps_per_round():
    # One worker, rows x0 = {0: 1} (y=+1), x1 = {1: 2} (y=-1), B = 1, tau = 2,
    # eta_k = 0.5 / (1 + k): eta_0 = 0.5 on row 0, eta_1 = 0.25 on row 1.
    # step 0: m = 0, y m = 0 < 1 -> r = -1, g = [-1, 0] -> w = [0.5, 0]
    # step 1: m = 2 * 0 = 0, y m = 0 < 1 -> r = +1, g = [0, 2] -> w = [0.5, -0.5]
    # with l2 = 0.2: step 1 scales w by (1 - 0.25 * 0.2) = 0.95 first: [0.475, -0.5]
    sh = inputs.SparseShards(d=2)
    sh.rowptr.append(np.array([0, 1, 2], np.int64))
    sh.col.append(np.array([0, 1], np.int32))
    sh.val.append(np.array([1.0, 2.0], np.float32))
    sh.y.append(np.array([1.0, -1.0], np.float32))
    sched = rounds.graph_schedule("identity", 1, 0)
    lr_at = lambda k: sgd.learning_rate("inverse", 0.5, 1.0, k)
    W, losses, _ = rounds.run_sparse(sh, 1, 1, "hinge", None, sched, tau=2, lr_at=lr_at)
    assert W[0] == pytest.approx([0.5, -0.5], abs=1e-15)
    assert losses[0] == pytest.approx(1.0, abs=1e-15)      # the last step's loss: max(0, 1 - 0)
    W, _, _ = rounds.run_sparse(sh, 1, 1, "hinge", None, sched, l2=0.2, tau=2, lr_at=lr_at)
    assert W[0] == pytest.approx([0.475, -0.5], abs=1e-15)


def test_local_steps_are_textbook_sgd_over_global_steps():
    sh = inputs.sparse_custom(seed=5, N=1, d=20, rows=60, max_len=8)
    B, tau, T, eta0, gamma = 10, 3, 4, 0.4, 0.2
    sched = rounds.graph_schedule("identity", 1, 0)
    lr_at = lambda k: sgd.learning_rate("inverse", eta0, gamma, k)
    Wo, _, _ = rounds.run_sparse(sh, T, B, "logistic", None, sched, tau=tau, lr_at=lr_at)
    Xd = np.zeros((60, 20))
    for r in range(60):
        a, b = sh.rowptr[0][r], sh.rowptr[0][r + 1]
        Xd[r, sh.col[0][a:b]] = sh.val[0][a:b]
    y = sh.y[0].astype(np.float64)
    w = np.zeros(20)
    for k in range(T * tau):                     # global step k: minibatch k mod 6, rate eta0 / (1 + gamma k)
        b0 = (k % 6) * B
        Xb, yb = Xd[b0:b0 + B], y[b0:b0 + B]
        s = 1.0 / (1.0 + np.exp(yb * (Xb @ w)))
        w = w - eta0 / (1.0 + gamma * k) / B * (Xb.T @ (-yb * s))
    assert Wo[0] == pytest.approx(w, abs=1e-14)


def test_hand_computed_softmax_step_reads_w_in_bf16():
    # C = 2 classes, d = 3, one row x = [1, 2, -1] (exact in bf16) of class 0,
    # B = 1, eta = 0.5.  W is not representable in bf16, so the logits use
    # RNE_bf16(W) while the update applies to the fp32 master:
    #   W[0] = [1 + 2^-8, 0.75 + 3 2^-10, -0.5 - 2^-11]
    #     -> [1 (tie, to even), 0.75 + 2^-8, -0.5]
    #   W[1] = [1 + 3 2^-8, -(2^-4 + 2^-13), 0.25 + 2^-10]
    #     -> [1 + 2^-6 (tie, to even), -2^-4, 0.25 (tie, to even)]
    # z = [1 + 1.5 + 2^-7 + 0.5, 1 + 2^-6 - 2^-3 - 0.25] = [3.0078125, 0.640625]
    # p1 = 1 / (1 + e^{2.3671875}) = 0.0857093..., p0 = 1 - p1
    # R = (p - e_0) / 1 = [p0 - 1, p1] = [-0.0857093..., 0.0857093...]; in bf16
    #   0.0857093 / 2^-11 = 175.53 -> 176 2^-11 = 0.0859375, so R = [-0.0859375, 0.0859375]
    # H[c] = W[c] - 0.5 R_c x:
    #   H[0] = W[0] + 0.04296875 [1, 2, -1] = [1.046875, 0.8388671875, -0.54345703125]
    #   H[1] = W[1] - 0.04296875 [1, 2, -1] = [0.96875, -0.1485595703125, 0.2939453125]
    # loss = ln(1 + e^{z1 - z0}) = log1p(exp(-2.3671875))
    W = np.array([[1 + 2 ** -8, 0.75 + 3 * 2 ** -10, -0.5 - 2 ** -11],
                  [1 + 3 * 2 ** -8, -(2 ** -4 + 2 ** -13), 0.25 + 2 ** -10]], np.float32)
    assert np.array_equal(W.astype(np.float64), [[1.00390625, 0.7529296875, -0.50048828125],
                                                 [1.01171875, -0.0626220703125, 0.2509765625]])
    Xbits = np.array([[0x3F80, 0x4000, 0xBF80]], np.uint16)       # bf16 bits of 1, 2, -1
    y = np.array([0], np.int32)
    H, loss = sgd.softmax_worker_step(W, Xbits, y, 0, 1, 0.5)
    assert H == pytest.approx(np.array([[1.046875, 0.8388671875, -0.54345703125],
                                        [0.96875, -0.1485595703125, 0.2939453125]]), abs=1e-15)
    assert loss == pytest.approx(math.log1p(math.exp(-2.3671875)), abs=1e-15)
    # The three plausible slips each move H: reading W unrounded, rounding the
    # master before the update, or skipping the bf16 rounding of R.
    Hu, _ = sgd.softmax_worker_step(W, Xbits, y, 0, 1, 0.5, mirror_bf16=False)
    assert np.abs(Hu - H).max() > 1e-4


def test_softmax_round_is_step_then_reduce_as_dense_matrices():
    # rounds.softmax_round against a restatement with dense matrices: per
    # worker the logits from the bf16-rounded model (torch's bf16 cast), the
    # softmax residual rounded to bf16, the fp32 master updated with an L2
    # term; then W' = P H with P written out, the mean loss and
    # ||W' - 1 wbar^T||_F.
    import torch
    N, d, C, B, t, lr, l2 = 3, 8, 4, 4, 1, 0.3, 0.05
    sh = inputs.dense_softmax(seed=5, N=N, d=d, C=C, rows=2 * B)
    rng = np.random.default_rng(2)
    W = (0.3 * rng.standard_normal((N, C * d))).astype(np.float32)
    nbr = np.array([[0, 2], [0, 1], [1, 2]])                 # ring: i <- i-1, weights 1/2
    wgt = np.full((3, 2), 0.5)
    P = np.zeros((3, 3))
    P[0, 0] = P[0, 2] = P[1, 0] = P[1, 1] = P[2, 1] = P[2, 2] = 0.5

    def bf16(a):
        return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).to(torch.float64).numpy()

    H = np.zeros((N, C * d))
    losses = []
    for i in range(N):
        X = bf16(np.asarray(torch.from_numpy(sh.X[i].view(np.int16)).view(torch.bfloat16).float()))[B:2 * B]
        yb = sh.y[i][B:2 * B]
        Wm = W[i].reshape(C, d).astype(np.float64)
        Z = X @ bf16(W[i].reshape(C, d)).T
        lse = np.logaddexp.reduce(Z, axis=1)
        losses.append(np.mean(lse - Z[np.arange(B), yb]))
        R = np.exp(Z - lse[:, None])
        R[np.arange(B), yb] -= 1.0
        R = bf16(R / B)
        H[i] = (Wm - lr * (R.T @ X + l2 * Wm)).reshape(-1)
    Wn = P @ H
    cons = np.sqrt(((Wn - Wn.mean(axis=0)) ** 2).sum())
    got, lval, c = rounds.softmax_round(W, sh, t, B, lr, nbr, wgt, l2=l2)
    assert got == pytest.approx(Wn, abs=1e-13)
    assert lval == pytest.approx(np.mean(losses), abs=1e-13)
    assert c == pytest.approx(cons, abs=1e-13)
