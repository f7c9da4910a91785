"""Pins for oracle/graphs.py and oracle/reduce.py against what the paper and
the mathematics fix (no GPU).

* SplitMix64 against the generator's published outputs.
* Fisher-Yates uniformity (brute force over all permutations of 3).
* Every graph kind: in-degree = out-degree = k+1, so P is doubly stochastic
  (Appendix A, "Network requirement").
* Spectral gap against the values printed in Fig. 2 / Section 6.1 and against
  circulant closed forms (Appendix A, "Spectral Gap").
* Mixing preserves the worker average; the consensus error contracts by at
  least sigma_2(P) per round (Appendix A's Perron-Frobenius bound).
"""
import cmath
import math
import os

import numpy as np
import pytest

from oracle import graphs, reduce, rounds

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_splitmix64_published_outputs():
    with open(os.path.join(GOLDEN, "splitmix64_seed0.txt")) as f:
        want = [int(l, 16) for l in f if l.strip() and not l.startswith("#")]
    rng = graphs.SplitMix64(0)
    assert [rng.next() for _ in want] == want


def test_uniform_range_and_rejection_limit():
    rng = graphs.SplitMix64(123)
    for m in (1, 2, 3, 7, 1000, (1 << 63) + 1):
        for _ in range(200):
            assert 0 <= rng.uniform(m) < m
    # m = 2^63 + 1: half of all 64-bit draws are rejected; values stay below m.
    counts = np.bincount([rng.uniform(7) for _ in range(70000)], minlength=7)
    chi2 = ((counts - 10000.0) ** 2 / 10000.0).sum()
    assert chi2 < 30.0          # 6 dof, p ~ 4e-5


def test_fisher_yates_uniform_over_all_permutations():
    rng = graphs.SplitMix64(7)
    seen = {}
    n = 60000
    for _ in range(n):
        p = tuple(graphs.fisher_yates(rng, 3))
        seen[p] = seen.get(p, 0) + 1
    assert len(seen) == 6        # a Sattolo-style off-by-one would give only the 2 cycles
    exp = n / 6.0
    chi2 = sum((c - exp) ** 2 / exp for c in seen.values())
    assert chi2 < 30.0


def _degrees(nbr):
    N = nbr.shape[0]
    indeg = np.array([len(set(r)) for r in nbr])
    outdeg = np.bincount(nbr.reshape(-1), minlength=N)
    return indeg, outdeg


@pytest.mark.parametrize("kind,N,k", [
    ("ring", 2, 1), ("ring", 17, 1), ("root", 4, 2), ("root", 25, 2), ("root", 32, 2), ("root", 256, 2),
    ("complete", 1, 0), ("complete", 8, 7), ("identity", 5, 0),
    ("random_regular", 2, 1), ("random_regular", 16, 2), ("random_regular", 64, 4), ("random_regular", 256, 4),
    ("random_regular", 9, 4), ("random_regular", 128, 8),
])
def test_graph_is_regular_and_doubly_stochastic(kind, N, k):
    for rnd in (0, 1, 5):
        nbr, wgt = graphs.build_graph(kind, N, k, graph_seed=99, rnd=rnd)
        assert nbr.shape == (N, k + 1)
        for i in range(N):
            assert i in nbr[i]
            assert list(nbr[i]) == sorted(set(nbr[i]))
        indeg, outdeg = _degrees(nbr)
        assert np.all(indeg == k + 1) and np.all(outdeg == k + 1)
        P = graphs.mixing_matrix(nbr, wgt)
        assert graphs.is_doubly_stochastic(P)


def test_random_regular_is_connected_and_seeded():
    for N, k in ((16, 2), (64, 4), (33, 3)):
        a, _ = graphs.build_graph("random_regular", N, k, graph_seed=5, rnd=3)
        b, _ = graphs.build_graph("random_regular", N, k, graph_seed=5, rnd=3)
        c, _ = graphs.build_graph("random_regular", N, k, graph_seed=5, rnd=4)
        assert np.array_equal(a, b) and not np.array_equal(a, c)
        # strong connectivity from node 0 along in-edges and along out-edges
        for edges in ("in", "out"):
            seen, stack = {0}, [0]
            while stack:
                u = stack.pop()
                nxt = a[u] if edges == "in" else [v for v in range(N) if u in a[v]]
                for v in nxt:
                    if v not in seen:
                        seen.add(v)
                        stack.append(int(v))
            assert len(seen) == N


def test_random_regular_rejects_infeasible():
    with pytest.raises(graphs.GraphError):
        graphs.build_graph("random_regular", 4, 4)        # k > N-1: no simple k-regular digraph
    with pytest.raises(graphs.GraphError):
        graphs.build_graph("random_regular", 4, 0)
    with pytest.raises(graphs.GraphError):
        graphs.build_graph("root", 3, 2)


def _gap_of(name, N):
    if name == "complete":
        A = np.ones((N, N))
    elif name == "directed_ring":
        A = np.eye(N) + np.roll(np.eye(N), -1, axis=1)      # i receives from i-1
    elif name == "directed_path":
        A = np.eye(N)
        for i in range(1, N):
            A[i, i - 1] = 1.0
    else:
        raise ValueError(name)
    return graphs.spectral_gap(graphs.adjacency_mixing(A))


def test_spectral_gaps_printed_in_paper():
    rows = []
    with open(os.path.join(GOLDEN, "spectral_gaps_paper.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                name, N, val, dec = line.split()[:4]
                rows.append((name, int(N), float(val), int(dec)))
    assert len(rows) == 5
    for name, N, val, dec in rows:
        assert round(_gap_of(name, N), dec) == pytest.approx(val), (name, N)


def _circulant_gap(offsets_weights, N):
    # P[i, (i - o) mod N] = w_o.  Circulant => normal => singular values are
    # the eigenvalue moduli |sum_o w_o exp(2 pi i o m / N)|.
    best = 0.0
    for m in range(1, N):
        lam = sum(w * cmath.exp(2j * math.pi * o * m / N) for o, w in offsets_weights)
        best = max(best, abs(lam))
    return 1.0 - best


@pytest.mark.parametrize("N", [4, 8, 16, 25, 32, 64, 128, 256])
def test_ring_and_root_gaps_match_circulant_closed_form(N):
    nbr, wgt = graphs.build_graph("ring", N, 1)
    gap = graphs.spectral_gap(graphs.mixing_matrix(nbr, wgt))
    assert gap == pytest.approx(1.0 - math.cos(math.pi / N), abs=1e-12)
    nbr, wgt = graphs.build_graph("root", N, 2)
    gap = graphs.spectral_gap(graphs.mixing_matrix(nbr, wgt))
    s = math.isqrt(N)
    assert gap == pytest.approx(_circulant_gap([(0, 1 / 3), (1, 1 / 3), (s, 1 / 3)], N), abs=1e-10)


def test_complete_gap_is_one_and_half_quarter_ring_is_one_half():
    nbr, wgt = graphs.build_graph("complete", 7, 6)
    assert graphs.spectral_gap(graphs.mixing_matrix(nbr, wgt)) == pytest.approx(1.0, abs=1e-12)
    nbr = np.array([[0, 1, 3], [0, 1, 2], [1, 2, 3], [0, 2, 3]])
    wgt = np.array([[0.5, 0.25, 0.25], [0.25, 0.5, 0.25], [0.25, 0.5, 0.25], [0.25, 0.25, 0.5]])
    P = graphs.mixing_matrix(nbr, wgt)
    assert graphs.is_doubly_stochastic(P)
    # eigenvalues 1/2 + 1/2 cos(2 pi m / 4) = {1, 1/2, 0, 1/2}
    assert graphs.spectral_gap(P) == pytest.approx(0.5, abs=1e-12)


def test_reduce_matches_explicit_small_case():
    # Hand check: 3 workers, d = 2, P rows {0:1/2, 1:1/2}, {1:1/2, 2:1/2}, {0:1/2, 2:1/2}
    H = np.array([[2.0, -4.0], [6.0, 0.0], [10.0, 8.0]])
    nbr = np.array([[0, 1], [1, 2], [0, 2]])
    wgt = np.full((3, 2), 0.5)
    W = reduce.stochastic_reduce(H, nbr, wgt)
    assert np.array_equal(W, np.array([[4.0, -2.0], [8.0, 4.0], [6.0, 2.0]]))
    # consensus error: mean row [6, 4/3]; deviations hand-summed
    dev = np.array([[-2.0, -10 / 3], [2.0, 8 / 3], [0.0, 2 / 3]])
    assert reduce.consensus_error(W) == pytest.approx(math.sqrt((dev ** 2).sum()), rel=1e-15)


@pytest.mark.parametrize("kind,N,k,regen", [("random_regular", 32, 4, True), ("root", 25, 2, False),
                                            ("ring", 16, 1, False), ("random_regular", 64, 2, True)])
def test_mixing_preserves_average_and_contracts_by_sigma2(kind, N, k, regen):
    rng = np.random.default_rng(1)
    W = rng.standard_normal((N, 50))
    sched = rounds.graph_schedule(kind, N, k, graph_seed=3, regenerate=regen)
    mean0 = W.mean(axis=0)
    E = reduce.consensus_error(W)
    for t in range(8):
        nbr, wgt = sched(t)
        P = graphs.mixing_matrix(nbr, wgt)
        s2 = 1.0 - graphs.spectral_gap(P)
        W = reduce.stochastic_reduce(W, nbr, wgt)
        En = reduce.consensus_error(W)
        assert En <= s2 * E * (1 + 1e-12) + 1e-12
        E = En
        assert np.allclose(W.mean(axis=0), mean0, atol=1e-13)


def test_complete_graph_reaches_consensus_in_one_round():
    W = np.random.default_rng(2).standard_normal((8, 30))
    _, cons = rounds.mixing_rounds(W, 2, rounds.graph_schedule("complete", 8, 7))
    assert cons[0] < 1e-13 and cons[1] < 1e-13


def test_simplex_bound_of_appendix_a():
    # ||P^t x - 1/n|| <= sigma_2^t for x in the probability simplex.
    N = 25
    nbr, wgt = graphs.build_graph("root", N, 2)
    P = graphs.mixing_matrix(nbr, wgt)
    s2 = 1.0 - graphs.spectral_gap(P)
    rng = np.random.default_rng(4)
    for _ in range(20):
        x = rng.random(N)
        x /= x.sum()
        v = x.copy()
        for t in range(1, 30):
            v = P @ v
            assert np.linalg.norm(v - 1.0 / N) <= s2 ** t + 1e-12


def test_matrix_form_of_the_reduce():
    # reduce_with_matrix: the hand case above, the complete graph's exact
    # column mean, and agreement with the per-row form on a random graph.
    H = np.array([[2.0, -4.0], [6.0, 0.0], [10.0, 8.0]])
    nbr = np.array([[0, 1], [1, 2], [0, 2]])
    P = graphs.mixing_matrix(nbr, np.full((3, 2), 0.5))
    assert np.array_equal(reduce.reduce_with_matrix(H, P), [[4.0, -2.0], [8.0, 4.0], [6.0, 2.0]])
    Hc = np.array([[1.0, 3.0], [5.0, -7.0], [0.0, 4.0], [2.0, 0.0]])     # column means 2 and 0
    nbr, wgt = graphs.build_graph("complete", 4, 3)
    assert np.array_equal(reduce.reduce_with_matrix(Hc, graphs.mixing_matrix(nbr, wgt)), [[2.0, 0.0]] * 4)
    rng = np.random.default_rng(7)
    Hr = rng.standard_normal((40, 30))
    nbr, wgt = graphs.build_graph("random_regular", 40, 4, 5, 2)
    assert np.allclose(reduce.reduce_with_matrix(Hr, graphs.mixing_matrix(nbr, wgt)),
                       reduce.stochastic_reduce(Hr, nbr, wgt), atol=1e-14)
