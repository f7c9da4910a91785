"""The graph-comparison study: its spectral gap against a closed form, its
smoothing, and (GPU) one short comparison run through the library."""
import math

import numpy as np
import pytest

from paper_1612_08608_gb300 import inputs
from paper_1612_08608_gb300.study import _smoothed, spectral_gap


def test_spectral_gap_closed_forms():
    N = 9
    # self weight 1/2, one in-neighbour i-1 with 1/2: P = (I + C)/2, a normal
    # circulant with singular values |1 + e^{2 pi i j / N}| / 2 = |cos(pi j / N)|
    nbr = np.array([[i, (i - 1) % N] for i in range(N)])
    wgt = np.full((N, 2), 0.5)
    assert spectral_gap(nbr, wgt) == pytest.approx(1.0 - math.cos(math.pi / N), abs=1e-12)
    # complete graph with equal weights: P = J / N, sigma_2 = 0
    nbr = np.array([list(range(N)) for _ in range(N)])
    assert spectral_gap(nbr, np.full((N, N), 1.0 / N)) == pytest.approx(1.0, abs=1e-12)


def test_smoothing_window():
    x = np.array([4.0, 2.0, 6.0, 0.0, 2.0])
    s = _smoothed(x, 2)
    assert np.isinf(s[0]) and s[1:].tolist() == [3.0, 4.0, 3.0, 1.0]


@pytest.mark.gpu
def test_graph_study_runs():
    from paper_1612_08608_gb300.study import compare
    sh = inputs.sparse_custom(seed=2, N=8, d=300, rows=8 * 16, max_len=20)
    res = compare(sh, "hinge", 16, 0.5, ref_rounds=16, max_rounds=64, chunk=8)
    assert [r["graph"] for r in res][0] == "complete" and res[0]["rounds_to_target"] == 16
    for r in res:
        assert r["bytes_per_worker_round"] == r["k"] * 300 * 4
        assert 0.0 < r["spectral_gap"] <= 1.0 + 1e-9
