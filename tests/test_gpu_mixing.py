"""GPU parity of the stochastic reduce alone (W <- P W, 20 rounds) against
the oracle: N in {8, 32, 128, 256}, d in {1e5, 1e6, 1e7}, k in {1, 2, 4,
N-1}.  At d = 1e5 every round is checked in full; above, the oracle follows
a seeded subset of 65,536 columns exactly (the reduce acts on each column on
its own) and the consensus error is checked against the Appendix A bound."""
import numpy as np
import pytest

from oracle import graphs, reduce, rounds
from paper_1612_08608_gb300 import inputs
from parity import rel_err_rows

pytestmark = pytest.mark.gpu

TOL = 1e-5


def _kind(N, k):
    return {1: "ring", N - 1: "complete"}.get(k, "random_regular")


def _ctx(N, d, k, regen=False):
    from paper_1612_08608_gb300 import Context
    ctx = Context(N, d, graph_seed=1, k=k)
    ctx.set_graph(_kind(N, k), regenerate=regen and _kind(N, k) == "random_regular")
    return ctx


@pytest.mark.parametrize("N", [8, 32, 128, 256])
@pytest.mark.parametrize("k", [1, 2, 4, "N-1"])
def test_mixing_every_round_d1e5(N, k):
    k = N - 1 if k == "N-1" else k
    d, T = 100000, 20
    W0 = inputs.mixing_params(seed=0, N=N, d=d)
    ctx = _ctx(N, d, k, regen=True)
    ctx.write_params(W0, 0)
    sched = rounds.graph_schedule(_kind(N, k), N, k, graph_seed=1, regenerate=_kind(N, k) == "random_regular")
    W_t = W0.astype(np.float64)
    for t in range(T):
        ctx.stochastic_reduce()
        W_n, _ = ctx.read_params()
        nbr, wgt = sched(t)
        ref = reduce.stochastic_reduce(W_t, nbr, wgt)
        assert rel_err_rows(W_n, ref) <= TOL, t
        loss, cons = ctx.read_metrics(t, 1)
        assert np.isnan(loss[0])
        cref = reduce.consensus_error(ref)
        assert abs(cons[0] - cref) <= 1e-4 * cref + 1e-6 * np.sqrt(N * d) * np.abs(ref).max(), (t, cons[0], cref)
        W_t = W_n.astype(np.float64)


@pytest.mark.parametrize("N,d,k", [(8, 1000000, 2), (32, 1000000, 4), (128, 1000000, 1), (256, 1000000, 255),
                                   (8, 10000000, 1), (32, 10000000, 2), (128, 10000000, 4), (256, 10000000, 4),
                                   (256, 10000000, 255)])
def test_mixing_large_column_subset(N, d, k):
    T = 20
    cols = np.sort(np.random.default_rng(N * 7 + k).choice(d, 65536, replace=False))
    W0 = inputs.mixing_params(seed=0, N=N, d=d)
    ctx = _ctx(N, d, k)
    ctx.write_params(W0, 0)
    del W0
    ctx.round(T)
    sched = rounds.graph_schedule(_kind(N, k), N, k, graph_seed=1)
    Wsub, _ = rounds.mixing_rounds(inputs.mixing_params(seed=0, N=N, d=d, cols=cols), T, sched)
    W_T, rnd = ctx.read_params()
    assert rnd == T
    assert rel_err_rows(W_T[:, cols], Wsub) <= 1e-4
    _, cons = ctx.read_metrics(0, T)
    nbr, wgt = sched(0)
    s2 = 1.0 - graphs.spectral_gap(graphs.mixing_matrix(nbr, wgt))
    prev = None
    for t in range(T):
        if prev is not None and prev > 1e-3 * cons[0]:
            assert cons[t] <= s2 * prev * (1 + 1e-4) + 1e-6 * cons[0], t
        prev = cons[t]
    full = reduce.consensus_error(W_T)
    assert abs(cons[T - 1] - full) <= 1e-3 * max(full, 1e-3 * cons[0])
