"""GPU parity of the sparse ASAP round (hinge / logistic SGD step, then the
stochastic reduce) against the CPU oracle, through the C ABI.

Protocol: each round is checked on its own, the oracle restarting from the
GPU's W_t (fp32 parameters within 1e-5 normwise relative error per worker);
the free-running loss trajectory must stay within 1e-4 absolute."""
import numpy as np
import pytest

from oracle import graphs, reduce, rounds
from paper_1612_08608_gb300 import inputs
from parity import rel_err_rows, sparse_round_matching

pytestmark = pytest.mark.gpu

TOL = 1e-5


def _ctx(N, d, k, seed, kind, regen, loss, B, lr, shards, explicit=None, residency="device", l2=0.0):
    from paper_1612_08608_gb300 import Context
    ctx = Context(N, d, graph_seed=seed, k=k)
    ctx.set_model(loss, batch=B, lr=lr, l2=l2)
    if explicit is not None:
        ctx.set_mixing(*explicit)
    else:
        ctx.set_graph(kind, regenerate=regen)
    ctx.set_shard_residency(residency)
    ctx.load_shards(shards)
    return ctx


def _run_parity(ctx, shards, T, B, loss, lr, sched, l2=0.0, check_graph=True, tau=1, lr_at=None):
    losses_gpu = []
    W_t, _ = ctx.read_params()
    for t in range(T):
        nbr, wgt = sched(t)
        if check_graph:
            g_nbr, _ = ctx.get_graph(t)
            assert np.array_equal(g_nbr, nbr)
        ctx.round(1)
        W_n, rnd = ctx.read_params()
        assert rnd == t + 1
        err, lref, cref = sparse_round_matching(W_t.astype(np.float64), W_n, shards, t, B, loss, lr, nbr, wgt,
                                                TOL, l2=l2, tau=tau, lr_at=lr_at)
        assert err <= TOL, (t, err)
        lg, cg = ctx.read_metrics(t, 1)
        assert abs(lg[0] - lref) <= 1e-5 * max(1.0, abs(lref)), (t, lg[0], lref)
        assert abs(cg[0] - cref) <= 1e-4 * cref + 1e-6 * np.abs(W_n).max() * np.sqrt(W_n.size), (t, cg[0], cref)
        losses_gpu.append(lg[0])
        W_t = W_n
    return np.array(losses_gpu)


def test_tiny_dense_logistic_ring_half_quarter():
    sh = inputs.tiny_dense_logistic(seed=0)
    N, B, lr, T = 4, 32, 0.1, 10
    nbr = np.array([[0, 1, 3], [0, 1, 2], [1, 2, 3], [0, 2, 3]], np.int32)
    wgt = np.array([[0.5, 0.25, 0.25], [0.25, 0.5, 0.25], [0.25, 0.5, 0.25], [0.25, 0.25, 0.5]], np.float32)
    sched = rounds.graph_schedule("explicit", N, 2, explicit=(nbr, wgt.astype(np.float64)))
    ctx = _ctx(N, sh.d, 2, 0, None, False, "logistic", B, lr, sh, explicit=(nbr, wgt))
    lg = _run_parity(ctx, sh, T, B, "logistic", lr, sched, check_graph=False)
    _, lref, _ = rounds.run_sparse(sh, T, B, "logistic", lr, sched)
    assert np.abs(lg - lref).max() <= 1e-4
    c = ctx.read_counters()
    assert c["reduces"] == N * T and c["consistent_inputs"] == N * 3 * T and c["timeouts"] == 0
    assert ctx.kernel_launches() == 2 * T + 1     # one gather of w at the first round


@pytest.mark.parametrize("loss", ["hinge", "logistic"])
@pytest.mark.parametrize("residency", ["device", "host"])
def test_ragged_edge_cases(loss, residency):
    # Empty rows, rows of up to 300 entries, a column in every row (runs much
    # longer than one 32-entry chunk), d not a multiple of 64, B not a
    # multiple of 32, a graph regenerated every round.
    N, d, B, lr, T = 6, 1000, 70, 0.5, 6
    rng = np.random.default_rng(5)
    lengths = [np.where(rng.random(4 * B) < 0.1, 0, rng.integers(1, 300, 4 * B)) for _ in range(N)]
    sh = inputs.sparse_custom(seed=11, N=N, d=d, rows=4 * B, lengths=lengths, hot_col=17)
    sched = rounds.graph_schedule("random_regular", N, 2, graph_seed=9, regenerate=True)
    ctx = _ctx(N, d, 2, 9, "random_regular", True, loss, B, lr, sh, residency=residency)
    _run_parity(ctx, sh, T, B, loss, lr, sched)


def test_all_empty_minibatch():
    # Minibatch 1 has no entries on any worker: margins 0, no column sums, the
    # loss of every row at m = 0.
    N, d, B, lr, T = 4, 300, 16, 0.5, 4
    rng = np.random.default_rng(21)
    lengths = [rng.integers(1, 20, 3 * B) for _ in range(N)]
    for ln in lengths:
        ln[B:2 * B] = 0
    sh = inputs.sparse_custom(seed=13, N=N, d=d, rows=3 * B, lengths=lengths)
    sched = rounds.graph_schedule("ring", N, 1)
    ctx = _ctx(N, d, 1, 0, "ring", False, "logistic", B, lr, sh)
    lg = _run_parity(ctx, sh, T, B, "logistic", lr, sched)
    assert abs(lg[1] - np.log(2.0)) <= 1e-6


def test_l2_regularised_logistic():
    N, d, B, lr, l2, T = 5, 300, 40, 0.3, 0.1, 5
    sh = inputs.sparse_custom(seed=4, N=N, d=d, rows=3 * B, max_len=30)
    sched = rounds.graph_schedule("ring", N, 1)
    ctx = _ctx(N, d, 1, 0, "ring", False, "logistic", B, lr, sh, l2=l2)
    _run_parity(ctx, sh, T, B, "logistic", lr, sched, l2=l2)


@pytest.mark.parametrize("B", [12288, 12289])
def test_large_minibatch(B):
    # Minibatches of more than 12,000 rows: many margin and column-sum CTAs
    # per worker, and column runs (the hot column is in every row) that span
    # hundreds of 32-entry chunks.
    N, d, lr, T = 3, 2000, 0.2, 2
    sh = inputs.sparse_custom(seed=12, N=N, d=d, rows=2 * B, max_len=12, hot_col=5)
    sched = rounds.graph_schedule("ring", N, 1)
    ctx = _ctx(N, d, 1, 0, "ring", False, "hinge", B, lr, sh)
    _run_parity(ctx, sh, T, B, "hinge", lr, sched)


@pytest.mark.parametrize("residency", ["device", "host"])
def test_local_steps_inverse_rate_l2(residency):
    # tau = 3 local steps per round (the intermediate updates and the L2
    # shrink kept as one scale until the reduce), eta_k = 0.5 / (1 + 0.1 k),
    # a graph regenerated every round.
    from oracle import sgd
    N, d, B, T, tau, l2 = 6, 1000, 32, 4, 3, 0.05
    sh = inputs.sparse_custom(seed=21, N=N, d=d, rows=10 * B, max_len=40, hot_col=3)
    sched = rounds.graph_schedule("random_regular", N, 2, graph_seed=4, regenerate=True)
    ctx = _ctx(N, d, 2, 4, "random_regular", True, "logistic", B, 0.5, sh, residency=residency, l2=l2)
    ctx.set_schedule(local_steps=tau, lr_schedule="inverse", gamma=0.1)
    lr_at = lambda k: sgd.learning_rate("inverse", 0.5, 0.1, k)
    lg = _run_parity(ctx, sh, T, B, "logistic", None, sched, l2=l2, tau=tau, lr_at=lr_at)
    _, lref, _ = rounds.run_sparse(sh, T, B, "logistic", None, sched, l2=l2, tau=tau, lr_at=lr_at)
    assert np.abs(lg - lref).max() <= 1e-4
    assert ctx.kernel_launches() == (3 * tau - 1) * T + 1    # local step, then update and gather but for the last


def test_inverse_rate_hinge_one_step():
    from oracle import sgd
    N, d, B, T = 5, 400, 24, 5
    sh = inputs.sparse_custom(seed=22, N=N, d=d, rows=4 * B, max_len=25)
    sched = rounds.graph_schedule("ring", N, 1)
    ctx = _ctx(N, d, 1, 0, "ring", False, "hinge", B, 0.8, sh)
    ctx.set_schedule(local_steps=1, lr_schedule="inverse", gamma=0.5)
    _run_parity(ctx, sh, T, B, "hinge", None, sched, lr_at=lambda k: sgd.learning_rate("inverse", 0.8, 0.5, k))


def test_schedule_argument_errors():
    from paper_1612_08608_gb300 import AsapError, Context
    ctx = Context(4, 256, graph_seed=0, k=1)
    ctx.set_model("softmax", batch=128, lr=0.1, num_classes=10)
    with pytest.raises(AsapError):
        ctx.set_schedule(local_steps=2)
    ctx.set_schedule(local_steps=1, lr_schedule="inverse", gamma=0.2)
    ctx.set_model("logistic", batch=16, lr=0.1)
    with pytest.raises(AsapError):
        ctx.set_schedule(local_steps=0)
    with pytest.raises(AsapError):
        ctx.set_schedule(local_steps=2, gamma=-1.0)


def test_single_worker_and_complete_graph():
    sh = inputs.sparse_custom(seed=6, N=1, d=200, rows=64, max_len=20)
    ctx = _ctx(1, 200, 0, 0, "identity", False, "hinge", 16, 0.2, sh)
    _run_parity(ctx, sh, 5, 16, "hinge", 0.2, rounds.graph_schedule("identity", 1, 0))
    sh = inputs.sparse_custom(seed=7, N=8, d=500, rows=64, max_len=20)
    ctx = _ctx(8, 500, 7, 0, "complete", False, "logistic", 16, 0.2, sh)
    _run_parity(ctx, sh, 4, 16, "logistic", 0.2, rounds.graph_schedule("complete", 8, 7))
    W, _ = ctx.read_params()
    assert np.abs(W - W[0]).max() <= 1e-6 * np.abs(W).max()


def test_sparse_hinge_svm_full_size():
    # RCV1-shaped: N=16, d=47,236, lognormal rows (mean 75), Zipf(1.1)
    # columns, hinge loss, B=256, k=2 random regular graph, 50 rounds.
    N, d, B, lr, T = 16, 47236, 256, 0.1, 50
    sh = inputs.sparse_hinge_svm(seed=0, N=N, rows=20000)
    sched = rounds.graph_schedule("random_regular", N, 2, graph_seed=0)
    ctx = _ctx(N, d, 2, 0, "random_regular", False, "hinge", B, lr, sh)
    lg = _run_parity(ctx, sh, T, B, "hinge", lr, sched)
    _, lref, _ = rounds.run_sparse(sh, T, B, "hinge", lr, sched)
    assert np.abs(lg - lref).max() <= 1e-4, np.abs(lg - lref).max()


def test_sparse_logistic_hashed_100_rounds():
    # The bench workload at its stated length: N=64, d=2^20, 50,000 rows per
    # worker with 100 uniform columns each, B=512 (97 minibatches, so rounds
    # 97-99 reuse the first three), k=4 expander drawn anew every round, 100
    # rounds.  The GPU runs free; every tenth round is also checked on its
    # own (the oracle restarted from the GPU's W_t, 1e-5), and the 100-round
    # loss trajectory must match the oracle's free-running one within 1e-4.
    N, d, B, lr, T = 64, 1 << 20, 512, 0.1, 100
    sh = inputs.sparse_logistic_hashed(seed=0, N=N, rows=50000)
    sched = rounds.graph_schedule("random_regular", N, 4, graph_seed=0, regenerate=True)
    ctx = _ctx(N, d, 4, 0, "random_regular", True, "logistic", B, lr, sh)
    for t in range(T):
        nbr, wgt = sched(t)
        assert np.array_equal(ctx.get_graph(t)[0], nbr)
        if t % 10 == 0:
            W_t, _ = ctx.read_params()
            ctx.round(1)
            W_n, rnd = ctx.read_params()
            assert rnd == t + 1
            err, lref, cref = sparse_round_matching(W_t.astype(np.float64), W_n, sh, t, B, "logistic", lr, nbr,
                                                    wgt, TOL)
            assert err <= TOL, (t, err)
            lg, cg = ctx.read_metrics(t, 1)
            assert abs(lg[0] - lref) <= 1e-5 * max(1.0, abs(lref)), (t, lg[0], lref)
            assert abs(cg[0] - cref) <= 1e-4 * cref + 1e-6 * np.abs(W_n).max() * np.sqrt(W_n.size), (t, cg[0], cref)
        else:
            ctx.round(1)
    lg, _ = ctx.read_metrics(0, T)
    del W_t, W_n
    _, lref, _ = rounds.run_sparse(sh, T, B, "logistic", lr, sched)
    assert np.abs(lg - lref).max() <= 1e-4, np.abs(lg - lref).max()
    assert ctx.read_counters()["timeouts"] == 0


def test_local_steps_full_shapes():
    # The bench's hashed workload with 4 local steps per round, eta_k =
    # 0.1 / (1 + 0.001 k) and a small L2 term: 2 rounds over 8 minibatches.
    from oracle import sgd
    N, d, B, T, tau, l2 = 64, 1 << 20, 512, 2, 4, 1e-4
    sh = inputs.sparse_logistic_hashed(seed=0, N=N, rows=tau * T * B)
    sched = rounds.graph_schedule("random_regular", N, 4, graph_seed=0, regenerate=True)
    ctx = _ctx(N, d, 4, 0, "random_regular", True, "logistic", B, 0.1, sh, l2=l2)
    ctx.set_schedule(local_steps=tau, lr_schedule="inverse", gamma=0.001)
    _run_parity(ctx, sh, T, B, "logistic", None, sched, l2=l2, tau=tau,
                lr_at=lambda k: sgd.learning_rate("inverse", 0.1, 0.001, k))


def test_local_steps_complete_graph_and_single_worker():
    # The complete graph's column-mean path and a lone worker (identity
    # graph) with the per-round L2 scale of several local steps.
    sh = inputs.sparse_custom(seed=23, N=8, d=500, rows=6 * 16, max_len=20)
    ctx = _ctx(8, 500, 7, 0, "complete", False, "logistic", 16, 0.3, sh, l2=0.05)
    ctx.set_schedule(local_steps=2)
    _run_parity(ctx, sh, 3, 16, "logistic", 0.3, rounds.graph_schedule("complete", 8, 7), l2=0.05, tau=2)
    W, _ = ctx.read_params()
    assert np.abs(W - W[0]).max() <= 1e-6 * np.abs(W).max()
    sh = inputs.sparse_custom(seed=24, N=1, d=300, rows=9 * 16, max_len=20)
    ctx = _ctx(1, 300, 0, 0, "identity", False, "logistic", 16, 0.3, sh, l2=0.05)
    ctx.set_schedule(local_steps=3)
    _run_parity(ctx, sh, 3, 16, "logistic", 0.3, rounds.graph_schedule("identity", 1, 0), l2=0.05, tau=3)


def test_notify_timeout_is_reported_and_recoverable():
    from paper_1612_08608_gb300 import AsapError
    sh = inputs.sparse_custom(seed=3, N=4, d=100, rows=64, max_len=10)
    ctx = _ctx(4, 100, 1, 0, "ring", False, "logistic", 16, 0.1, sh)
    ctx.round(1)
    W1, _ = ctx.read_params()
    ctx.set_wait_limit_ns(20_000_000)         # 20 ms
    ctx.debug_skip_notify(2)                  # worker 2 never publishes NOTIFY
    ctx.round(1)
    with pytest.raises(AsapError) as ei:
        ctx.sync()
    assert ei.value.name == "ASAP_ERR_TIMEOUT"
    assert ctx.read_counters()["timeouts"] >= 1
    # Resume from the last good parameters: the protocol state is reset.
    ctx.write_params(W1, 1)
    ctx.round(2)
    W3, rnd = ctx.read_params()
    assert rnd == 3 and np.isfinite(W3).all()


@pytest.mark.parametrize("residency", ["device", "host"])
def test_lagged_metric_reads_match_a_full_sync(residency):
    # Round t's metrics read while round t+1 runs (the read waits for round t
    # only) equal those read after a full drain.
    sh = inputs.sparse_custom(seed=12, N=8, d=3000, rows=256, max_len=60, hot_col=3)
    ctx = _ctx(8, 3000, 2, 4, "random_regular", True, "logistic", 64, 0.3, sh, residency=residency)
    T = 7
    lagged = []
    for t in range(T):
        ctx.round(1)
        if t > 0:
            lagged.append(ctx.read_metrics(t - 1, 1))
    lagged.append(ctx.read_metrics(T - 1, 1))
    ctx.sync()
    loss, cons = ctx.read_metrics(0, T)
    assert np.array_equal(np.concatenate([m[0] for m in lagged]), loss)
    assert np.array_equal(np.concatenate([m[1] for m in lagged]), cons)
    assert np.isfinite(loss).all() and np.isfinite(cons).all()


def test_lagged_metric_read_reports_a_timeout():
    from paper_1612_08608_gb300 import AsapError
    sh = inputs.sparse_custom(seed=3, N=4, d=100, rows=64, max_len=10)
    ctx = _ctx(4, 100, 1, 0, "ring", False, "logistic", 16, 0.1, sh)
    ctx.round(1)
    W1, _ = ctx.read_params()
    ctx.set_wait_limit_ns(20_000_000)         # 20 ms
    ctx.debug_skip_notify(1)
    ctx.round(1)
    with pytest.raises(AsapError) as ei:
        ctx.read_metrics(1, 1)
    assert ei.value.name == "ASAP_ERR_TIMEOUT"
    ctx.write_params(W1, 1)
    ctx.round(1)
    loss, cons = ctx.read_metrics(1, 1)
    assert np.isfinite(loss).all() and np.isfinite(cons).all()


def test_two_runs_bit_identical():
    sh = inputs.sparse_custom(seed=8, N=8, d=3000, rows=256, max_len=60, hot_col=3)
    outs = []
    for _ in range(2):
        ctx = _ctx(8, 3000, 2, 5, "random_regular", True, "hinge", 64, 0.3, sh)
        ctx.round(8)
        outs.append(ctx.read_params()[0])
        ctx.close()
    assert np.array_equal(outs[0], outs[1])
