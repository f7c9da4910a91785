"""The library's minibatch index builder (host only, no GPU): the image that
asap_load_shards uploads, decoded and checked against a plain restatement
from the shards -- padded rows, list positions, the (column, row)-sorted
copy of the entries, and the slab-major list of distinct (worker, column)
pairs with its padded slab regions."""
import numpy as np
import pytest

from paper_1612_08608_gb300 import inputs
from paper_1612_08608_gb300.api import AsapError, debug_batch_image

PAD = 0xFFFFFFFF


def _view(img, off, dtype, n):
    return np.frombuffer(img[off:off + np.dtype(dtype).itemsize * n].tobytes(), dtype=dtype)


@pytest.mark.parametrize("S", [64, 1024])
def test_batch_image_matches_the_shards(S):
    N, d, B, t = 3, 1000, 20, 1
    rng = np.random.default_rng(8)
    lengths = [np.where(rng.random(3 * B) < 0.15, 0, rng.integers(1, 40, 3 * B)) for _ in range(N)]
    sh = inputs.sparse_custom(seed=31, N=N, d=d, rows=3 * B, lengths=lengths, hot_col=7)
    img, desc, (list_off, soff_off, list_len) = debug_batch_image(sh, B, S, t)
    n_slabs = -(-((d + 63) // 64 * 64) // S)
    lst = _view(img, list_off, np.uint32, list_len)
    soff = _view(img, soff_off, np.int32, n_slabs + 1)
    assert soff[0] == 0 and soff[-1] == list_len and np.all(np.diff(soff) % 4 == 0)

    pairs = set()
    for i in range(N):
        rp_o, y_o, pw_o, val_o, cp_o, cv_o, cr_o, nnz_pad, nnz = (int(v) for v in desc[i])
        rp = _view(img, rp_o, np.int32, B + 1)
        pw = _view(img, pw_o, np.int32, nnz_pad)
        vals = _view(img, val_o, np.float32, nnz_pad)
        r0 = t * B
        entries = []                                   # (col, row, val, padded index)
        for b in range(B):
            a, e = sh.rowptr[i][r0 + b], sh.rowptr[i][r0 + b + 1]
            n = e - a
            assert rp[b + 1] - rp[b] == -(-n // 4) * 4 and rp[b] % 4 == 0
            for j in range(n):
                c = int(sh.col[i][a + j])
                q = rp[b] + j
                assert vals[q] == sh.val[i][a + j]
                p = int(pw[q])
                assert lst[p] == (i << 16) | (c % S) and soff[c // S] <= p < soff[c // S + 1]
                entries.append((c, b, sh.val[i][a + j], q))
                pairs.add((i, c))
            assert np.all(vals[rp[b] + n:rp[b + 1]] == 0)
        assert rp[B] == nnz_pad and len(entries) == nnz
        assert np.array_equal(_view(img, y_o, np.float32, B), sh.y[i][r0:r0 + B])
        # the (column, row)-sorted copy
        entries.sort(key=lambda x: (x[0], x[1]))
        cp = _view(img, cp_o, np.int32, nnz)
        cv = _view(img, cv_o, np.float32, nnz)
        cr = _view(img, cr_o, np.uint16, nnz)
        assert np.array_equal(cr, [x[1] for x in entries])
        assert np.array_equal(cv, np.array([x[2] for x in entries], np.float32))
        assert np.array_equal(cp, [pw[x[3]] for x in entries])

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
