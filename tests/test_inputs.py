"""The seeded synthetic workloads follow their stated recipes: shapes,
row-length and column-popularity distributions, value distributions, row
normalisation, label noise, and per-worker seeding.  No GPU."""
import numpy as np
import pytest

from paper_1612_08608_gb300 import inputs


def _teacher(seed, d):
    return inputs._rng(seed, inputs._TEACHER).standard_normal(d)


def _row_scores(sh, i, wstar):
    rp, col, val = sh.rowptr[i], sh.col[i], sh.val[i]
    row_of = np.repeat(np.arange(rp.shape[0] - 1), np.diff(rp))
    return np.bincount(row_of, weights=val.astype(np.float64) * wstar[col], minlength=rp.shape[0] - 1)


def _agreement(sh, seed):
    """Share of labels equal to the teacher's sign (1 - flip rate)."""
    wstar = _teacher(seed, sh.d)
    agree = [np.mean(np.where(_row_scores(sh, i, wstar) >= 0, 1.0, -1.0) == sh.y[i]) for i in range(sh.N)]
    return float(np.mean(agree))


def _check_csr(sh):
    for i in range(sh.N):
        rp, col = sh.rowptr[i], sh.col[i]
        assert rp[0] == 0 and np.all(np.diff(rp) >= 0) and rp[-1] == col.shape[0] == sh.val[i].shape[0]
        assert col.dtype == np.int32 and sh.val[i].dtype == np.float32 and sh.y[i].dtype == np.float32
        assert col.min() >= 0 and col.max() < sh.d
        assert set(np.unique(sh.y[i])) <= {-1.0, 1.0}
        # distinct, ascending ids within every row
        inner = np.ones(col.shape[0], dtype=bool)
        inner[rp[:-1][np.diff(rp) > 0]] = False
        assert np.all(np.diff(col.astype(np.int64))[inner[1:]] > 0)


def test_tiny_dense_logistic_recipe():
    sh = inputs.tiny_dense_logistic(seed=0)
    _check_csr(sh)
    assert sh.N == 4 and sh.d == 64 and all(sh.n_rows(i) == 256 for i in range(4))
    for i in range(4):
        assert np.all(np.diff(sh.rowptr[i]) == 64)
    v = np.concatenate(sh.val)
    assert abs(v.mean()) < 0.02 and abs(v.std() - 1.0) < 0.02
    assert abs((1.0 - _agreement(sh, 0)) - 0.05) < 0.025          # 5 % flipped labels


def test_sparse_hinge_svm_recipe():
    N, rows = 2, 4000
    sh = inputs.sparse_hinge_svm(seed=3, N=N, rows=rows)
    _check_csr(sh)
    assert sh.d == 47236
    lengths = np.concatenate([np.diff(sh.rowptr[i]) for i in range(N)])
    assert lengths.min() >= 5 and lengths.max() <= 1000
    assert 70.0 < lengths.mean() < 80.0                            # lognormal with mean 75
    assert 0.6 < np.mean(lengths < 75) < 0.8                       # lognormal, sigma 1: P(L < mean) = Phi(1/2)
    col = np.concatenate(sh.col)
    # Zipf popularity over ranks: column 0 in nearly every row, frequencies
    # falling with the column id.
    freq = np.bincount(col, minlength=sh.d)
    assert freq[0] > 0.9 * N * rows
    assert freq[:10].sum() > freq[100:110].sum() > freq[10000:10010].sum()
    val = np.concatenate(sh.val)
    assert val.min() > 0.0
    for i in range(N):
        rp = sh.rowptr[i]
        row_of = np.repeat(np.arange(rows), np.diff(rp))
        norms = np.sqrt(np.bincount(row_of, weights=sh.val[i].astype(np.float64) ** 2, minlength=rows))
        assert np.allclose(norms, 1.0, atol=1e-5)
    assert abs((1.0 - _agreement(sh, 3)) - 0.03) < 0.012           # 3 % flipped labels


def test_sparse_logistic_hashed_recipe():
    N, rows = 2, 3000
    sh = inputs.sparse_logistic_hashed(seed=4, N=N, rows=rows)
    _check_csr(sh)
    assert sh.d == 1 << 20
    for i in range(N):
        assert np.all(np.diff(sh.rowptr[i]) == 100)
    col = np.concatenate(sh.col)
    buckets = np.bincount(col >> 16, minlength=16)                  # 16 equal ranges of the hashed space
    expect = col.shape[0] / 16
    assert np.all(np.abs(buckets - expect) < 0.03 * expect)
    v = np.concatenate(sh.val)
    assert abs(v.mean()) < 0.01 and abs(v.std() - 1.0) < 0.01
    assert abs((1.0 - _agreement(sh, 4)) - 0.03) < 0.012


def test_dense_softmax_recipe():
    pytest.importorskip("torch")
    d, C, rows = 256, 10, 4096
    sh = inputs.dense_softmax(seed=5, N=1, d=d, C=C, rows=rows)
    X, y = sh.X[0], sh.y[0]
    assert X.dtype == np.uint16 and X.shape == (rows, d) and y.dtype == np.int32 and y.shape == (rows,)
    x = inputs.bf16_bits_to_f32(X).astype(np.float64)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    assert y.min() >= 0 and y.max() < C
    share = np.bincount(y, minlength=C) / rows
    assert share.min() > 0.04 and share.max() < 0.2                 # logits ~ N(0, 1): no class dominates
    # Labels are Gumbel-perturbed argmaxes of the teacher's logits: the
    # noiseless argmax wins far more often than chance (1 / C).
    Wstar = (inputs._rng(5, inputs._TEACHER).standard_normal((C, d)) / np.sqrt(d))
    assert np.mean(np.argmax(x @ Wstar.T, axis=1) == y) > 0.25


def test_workers_are_seeded_independently():
    a = inputs.sparse_logistic_hashed(seed=9, N=2, d=4096, rows=64, nnz=10)
    b = inputs.sparse_logistic_hashed(seed=9, N=3, d=4096, rows=64, nnz=10)
    c = inputs.sparse_logistic_hashed(seed=10, N=2, d=4096, rows=64, nnz=10)
    for i in range(2):                                              # worker i does not depend on N
        assert np.array_equal(a.col[i], b.col[i]) and np.array_equal(a.val[i], b.val[i])
        assert np.array_equal(a.y[i], b.y[i])
    assert not np.array_equal(a.col[0], a.col[1])
    assert not np.array_equal(a.col[0], c.col[0])
    full = inputs.mixing_params(2, 5, 300)
    cols = np.array([0, 7, 299])
    assert np.array_equal(inputs.mixing_params(2, 5, 300, rows=range(1, 3)), full[1:3])
    assert np.array_equal(inputs.mixing_params(2, 5, 300, cols=cols), full[:, cols])
