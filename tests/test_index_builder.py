"""The library's minibatch index builder (host only, no GPU): the image that
asap_load_shards uploads, decoded and checked against a plain restatement
from the shards -- the (column, row)-sorted entries with their list
positions, the margin segments' slots and the rows of their slots, the
column-sum ranges cut at column boundaries, and the slab-major list of
distinct (worker, column) pairs with its padded slab regions."""
import numpy as np
import pytest

from paper_1612_08608_gb300 import inputs
from paper_1612_08608_gb300.api import AsapError, debug_batch_image

PAD = 0xFFFFFFFF


def _view(img, off, dtype, n):
    return np.frombuffer(img[off:off + np.dtype(dtype).itemsize * n].tobytes(), dtype=dtype)


@pytest.mark.parametrize("S,Q,max_len", [(64, 1, 40), (1024, 3, 40), (64, 8, 400)])
def test_batch_image_matches_the_shards(S, Q, max_len):
    # max_len 400 with B = 20 rows: about 3,400 entries, so minibatches span
    # more than one 256-entry margin segment and 1024-entry tile
    N, d, B, t = 3, 1000, 20, 1
    rng = np.random.default_rng(8)
    lengths = [np.where(rng.random(3 * B) < 0.15, 0, rng.integers(1, max_len, 3 * B)) for _ in range(N)]
    sh = inputs.sparse_custom(seed=31, N=N, d=d, rows=3 * B, lengths=lengths, hot_col=7)
    _check_image(sh, N, d, B, S, Q, t)


def test_batch_image_edge_cases():
    N, d, B = 4, 777, 16
    rows = 3 * B
    z = np.zeros(rows, np.int64)
    # worker 0: an empty minibatch at t = 1 between non-empty ones; worker 1:
    # three entries for eight CTAs (empty column-sum ranges); worker 2: every
    # row of window 1 holds the same single column; worker 3: full rows
    l0 = np.full(rows, 5)
    l0[B:2 * B] = 0
    l1 = z.copy()
    l1[[B + 1, B + 7, B + 15]] = 1
    l2 = np.full(rows, 1)
    l3 = np.full(rows, 60)
    sh = inputs.sparse_custom(seed=5, N=N, d=d, rows=rows, lengths=[l0, l1, l2, l3])
    for r in range(B, 2 * B):                  # worker 2: column 3 in every row of window 1
        sh.col[2][sh.rowptr[2][r]] = 3
    for S, Q, t in [(8, 8, 1), (8, 1, 1), (1024, 8, 1), (64, 2, 2), (16, 5, 0)]:
        _check_image(sh, N, d, B, S, Q, t)


def _check_image(sh, N, d, B, S, Q, t):
    img, desc, (list_off, soff_off, list_len) = debug_batch_image(sh, B, S, t, ctas_per_worker=Q)
    n_slabs = -(-((d + 63) // 64 * 64) // S)
    lst = _view(img, list_off, np.uint32, list_len)
    soff = _view(img, soff_off, np.int32, n_slabs + 1)
    assert soff[0] == 0 and soff[-1] == list_len and np.all(np.diff(soff) % 4 == 0)

    pairs = set()
    for i in range(N):
        y_o, cp_o, cv_o, cr_o, cs_o, bd_o, nnz, zero = (int(v) for v in desc[i])
        assert zero == 0
        r0 = t * B
        entries = []                                   # (col, row, val)
        for b in range(B):
            a, e = sh.rowptr[i][r0 + b], sh.rowptr[i][r0 + b + 1]
            for j in range(e - a):
                c = int(sh.col[i][a + j])
                entries.append((c, b, sh.val[i][a + j]))
                pairs.add((i, c))
        assert len(entries) == nnz
        assert np.array_equal(_view(img, y_o, np.float32, B), sh.y[i][r0:r0 + B])
        # the (column, row)-sorted entries: value, row, and the list position
        # of the entry's (worker, column) pair
        entries.sort(key=lambda x: (x[0], x[1]))
        cp = _view(img, cp_o, np.int32, nnz)
        cv = _view(img, cv_o, np.float32, nnz)
        cr = _view(img, cr_o, np.uint16, nnz)
        assert np.array_equal(cr, [x[1] for x in entries])
        assert np.array_equal(cv, np.array([x[2] for x in entries], np.float32))
        for e, (c, _, _) in enumerate(entries):
            p = int(cp[e])
            assert lst[p] == (i << 16) | (c % S) and soff[c // S] <= p < soff[c // S + 1]
        # margin segments of 256 entries: slots numbered row by row, by
        # column within a row
        cs = _view(img, cs_o, np.uint16, nnz)
        for e0 in range(0, nnz, 256):
            e1 = min(e0 + 256, nnz)
            seg = sorted(range(e0, e1), key=lambda e: (entries[e][1], entries[e][0]))
            assert [int(cs[e]) for e in seg] == list(range(e1 - e0))
        # column-sum ranges: cut at the first column boundary at or after q nnz / Q
        bd = _view(img, bd_o, np.int32, Q + 1)
        assert bd[0] == 0 and bd[Q] == nnz and np.all(np.diff(bd) >= 0)
        for q in range(1, Q):
            e = int(bd[q])
            assert e >= q * nnz // Q
            assert e == 0 or e == nnz or entries[e][0] != entries[e - 1][0]
            assert all(entries[x][0] == entries[x - 1][0] for x in range(max(q * nnz // Q, 1), e))

    # every slab region: the distinct (worker, column) pairs of its columns,
    # by worker then column, padded at the end
    for s in range(n_slabs):
        region = lst[soff[s]:soff[s + 1]]
        want = sorted((i, c) for (i, c) in pairs if c // S == s)
        real = region[region != PAD]
        assert np.all(region[len(real):] == PAD) and len(region) - len(real) < 4
        assert [(int(v) >> 16, s * S + (int(v) & 0xFFFF)) for v in real] == want


def test_batch_image_rejects_bad_slab_width():
    sh = inputs.sparse_custom(seed=1, N=2, d=100, rows=16, max_len=5)
    with pytest.raises(AsapError):
        debug_batch_image(sh, 8, 48, 0)


def test_batch_image_rejects_a_minibatch_past_the_shard():
    sh = inputs.sparse_custom(seed=1, N=2, d=100, rows=16, max_len=5)
    with pytest.raises(ValueError):
        debug_batch_image(sh, 8, 64, 2)
