"""The graph-comparison study of bench.py (Section 6.1): its target rule,
first-crossing search, sigma_2 and hinge evaluation on cases with a known
answer (no GPU)."""
import math
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def test_target_is_ninety_percent_of_the_drop():
    # drop from 1.0 to a lowest value of 0.5: 90 % of it is reached at 0.55
    assert bench.study_target(1.0, [1.0, 0.6, 0.5, 0.52]) == pytest.approx(0.55)
    assert bench.study_target(2.0, [2.0, 1.0], frac=0.5) == pytest.approx(1.5)


def test_first_reaching():
    xs, fs = [0, 10, 20, 30], [1.0, 0.6, 0.55, 0.5]
    assert bench.first_reaching(xs, fs, 0.55) == 20
    assert bench.first_reaching(xs, fs, 0.4) is None
    assert bench.first_reaching(xs, fs, 2.0) == 0


def test_sigma2_closed_forms():
    N = 9
    # self weight 1/2 and i-1 with 1/2: singular values |cos(pi j / N)|
    nbr = np.array([[i, (i - 1) % N] for i in range(N)])
    assert bench.sigma2(nbr, np.full((N, 2), 0.5)) == pytest.approx(math.cos(math.pi / N), abs=1e-12)
    nbr = np.array([list(range(N)) for _ in range(N)])
    assert bench.sigma2(nbr, np.full((N, N), 1.0 / N)) == pytest.approx(0.0, abs=1e-12)


def test_hinge_evaluation_by_hand():
    # rows {0: 1}, {1: 2, 2: -1}, {} with labels +1, -1, +1 at w = [0.5, 1, 0]:
    # margins 0.5, 2, 0 -> hinge 0.5, 3, 1 -> mean 1.5
    rowptr = np.array([0, 1, 3, 3])
    col = np.array([0, 1, 2])
    val = np.array([1.0, 2.0, -1.0], np.float32)
    y = np.array([1.0, -1.0, 1.0], np.float32)
    assert bench.hinge_loss_at(np.array([0.5, 1.0, 0.0]), rowptr, col, val, y) == pytest.approx(1.5)
