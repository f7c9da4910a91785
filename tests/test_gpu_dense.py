"""GPU parity of the dense softmax-regression round (tcgen05 bf16 GEMMs with
fp32 accumulation, softmax across a cluster, fp32 master update, then the
stochastic reduce writing the next round's bf16 copy) against the oracle,
which mirrors the bf16 rounding points.  Tolerance: 1e-3 normwise relative
error per worker per round (bf16-input GEMM path), loss within 1e-4."""
import numpy as np
import pytest

from oracle import rounds, sgd
from paper_1612_08608_gb300 import inputs
from parity import rel_err_rows

pytestmark = pytest.mark.gpu

TOL = 1e-3


def _run(N, d, C, B, lr, k, kind, T, seed=0, l2=0.0, w0_scale=0.0, gamma=None):
    from paper_1612_08608_gb300 import Context
    sh = inputs.dense_softmax(seed=seed, N=N, d=d, C=C, rows=T * B)
    ctx = Context(N, d, graph_seed=seed, k=k)
    ctx.set_model("softmax", batch=B, lr=lr, num_classes=C, l2=l2)
    ctx.set_graph(kind)
    if gamma is not None:
        ctx.set_schedule(local_steps=1, lr_schedule="inverse", gamma=gamma)
    ctx.load_dense_shards(sh)
    sched = rounds.graph_schedule(kind, N, k, graph_seed=seed)
    W_t, _ = ctx.read_params()
    assert W_t.shape == (N, C * d) and not W_t.any()
    if w0_scale:
        W_t = (w0_scale * np.random.default_rng(seed).standard_normal(W_t.shape)).astype(np.float32)
        ctx.write_params(W_t, 0)
    for t in range(T):
        ctx.round(1)
        W_n, rnd = ctx.read_params()
        assert rnd == t + 1
        nbr, wgt = sched(t)
        eta = lr if gamma is None else sgd.learning_rate("inverse", lr, gamma, t)
        ref, lref, cref = rounds.softmax_round(W_t, sh, t, B, eta, nbr, wgt, l2=l2)
        err = rel_err_rows(W_n, ref)
        assert err <= TOL, (t, err)
        lg, cg = ctx.read_metrics(t, 1)
        assert abs(lg[0] - lref) <= 1e-4 * max(1.0, abs(lref)), (t, lg[0], lref)
        assert abs(cg[0] - cref) <= 2e-3 * cref + 1e-7, (t, cg[0], cref)
        W_t = W_n
    return ctx


def test_dense_small_one_cluster_cta():
    _run(N=4, d=256, C=10, B=128, lr=0.5, k=1, kind="ring", T=3)


def test_dense_ragged_classes_two_cluster_ctas_l2():
    _run(N=6, d=512, C=300, B=256, lr=0.3, k=2, kind="random_regular", T=3, seed=2, l2=0.01)


@pytest.mark.parametrize("C,B", [(600, 256), (1024, 384)])
def test_dense_cluster_geometries(C, B):
    # Forward clusters of three CTAs (C=600) and of four full class tiles
    # with an odd number of row tiles (C=1024, B=384).  Random initial
    # parameters: from W = 0, every class absent from the first minibatch
    # gets the same row, their logits and residuals in the next round are
    # exactly equal, and one fp32-versus-fp64 rounding decision at the bf16
    # cast of R moves hundreds of them together by one bf16 ulp (a CPU
    # restatement in the kernel's fp32 order differs from the oracle by
    # 3.7e-3 there, as the GPU does).
    _run(N=3, d=256, C=C, B=B, lr=0.2, k=1, kind="ring", T=2, seed=3, w0_scale=0.05)


def test_dense_inverse_rate_l2():
    # eta_t = 0.5 / (1 + 0.5 t) on the dense path (one local step per round)
    _run(N=4, d=256, C=20, B=128, lr=0.5, k=1, kind="ring", T=4, seed=4, l2=0.02, gamma=0.5)


def test_dense_softmax_full_size():
    # N=32 workers, d=2048 bf16 features, C=1000 classes, B=512, root graph.
    ctx = _run(N=32, d=2048, C=1000, B=512, lr=0.1, k=2, kind="root", T=3)
    assert ctx.read_counters()["timeouts"] == 0
