"""Communication graphs and mixing matrices (oracle; test infrastructure only).

Paper passages followed:
* Section 3.1 and Fig. 2: the all-reduce (complete) graph, the chain graph,
  and the "root" expander in which node i sends to i+1 and to i+sqrt(N).
* Section 3.1 (such graphs are cheap to build, so a failed node can be
  routed around by building a new one): a graph is produced from a seed,
  and may be produced anew every round.
* Appendix A, "Network requirement": A_ij = 1 iff (j, i) is an edge, self
  included; P = diag(d_in)^-1 A; P must be doubly stochastic, i.e. every node
  has the same in- and out-degree.
* Appendix A, "Spectral Gap": gap = 1 - sigma_2(P), sigma_2 the second
  largest *singular* value.

The paper does not say how a random expander is drawn.  The reading used
here (and stated in the design notes) is:

* PRNG: SplitMix64 (Steele, Lea & Flood, OOPSLA 2014), state advanced by the
  golden gamma 0x9E3779B97F4A7C15 and mixed by the "variant 13" finaliser.
  Round r starts from ``graph_seed XOR (gamma * (r + 1) mod 2^64)``;
  a graph that is not regenerated uses r = 0.
* ``uniform(m)``: draw v; reject while v >= 2^64 - (2^64 mod m); return v mod m.
* Fisher-Yates: start from the identity, for t = N-1 .. 1 swap slots t and
  uniform(t+1).
* random k-regular: (1) a random permutation pi gives a Hamiltonian cycle,
  node pi[(t+1) mod N] receiving from pi[t] (so the graph is connected);
  (2) k-1 more layers.  Each layer draws permutations sigma by Fisher-Yates
  until one is admissible: sigma[i] != i and sigma[i] not already an
  in-neighbour of i, for every i (node i then receives from sigma[i]).
  Slot t is final right after step t of the shuffle, so a draw is abandoned
  at the first inadmissible slot (slot 0 is checked after the loop); this
  rejection sampler is exact (uniform over admissible permutations) and
  only cheaper than checking whole permutations.  At most 100,000 draws
  per layer.
* Each row lists {i} and its in-neighbours in ascending order, with equal
  weights 1/(k+1) (Eq. A.1's equal-weight average).
"""
from __future__ import annotations

import math

import numpy as np

GOLDEN_GAMMA = 0x9E3779B97F4A7C15
_MASK = (1 << 64) - 1
MAX_LAYER_TRIES = 100000


class GraphError(ValueError):
    """Raised when a graph of the requested kind cannot be built."""


class SplitMix64:
    """SplitMix64 as published by Steele, Lea & Flood (2014)."""

    def __init__(self, state: int):
        self.state = state & _MASK

    def next(self) -> int:
        self.state = (self.state + GOLDEN_GAMMA) & _MASK
        z = self.state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK
        return z ^ (z >> 31)

    def uniform(self, m: int) -> int:
        """Unbiased integer in [0, m) by rejection of the top partial block."""
        if m <= 0:
            raise ValueError("m must be positive")
        limit = (1 << 64) - ((1 << 64) % m)
        while True:
            v = self.next()
            if v < limit:
                return v % m


def round_state(graph_seed: int, rnd: int) -> int:
    return (graph_seed ^ ((GOLDEN_GAMMA * (rnd + 1)) & _MASK)) & _MASK


def fisher_yates(rng: SplitMix64, n: int) -> list:
    perm = list(range(n))
    for t in range(n - 1, 0, -1):
        j = rng.uniform(t + 1)
        perm[t], perm[j] = perm[j], perm[t]
    return perm


def _rows_from_in_neighbours(in_nbrs) -> np.ndarray:
    return np.array([sorted({i} | set(s)) for i, s in enumerate(in_nbrs)], dtype=np.int64)


def ring_graph(N: int) -> np.ndarray:
    """Chain closed into a directed ring: node i receives from i-1."""
    if N < 2:
        raise GraphError("ring needs N >= 2")
    return _rows_from_in_neighbours([{(i - 1) % N} for i in range(N)])


def root_graph(N: int) -> np.ndarray:
    """Section 3.1 root expander: i sends to i+1 and i+isqrt(N), so i
    receives from i-1 and i-isqrt(N)."""
    s = math.isqrt(N)
    if N < 4:
        raise GraphError("root graph needs N >= 4 (isqrt(N) >= 2)")
    return _rows_from_in_neighbours([{(i - 1) % N, (i - s) % N} for i in range(N)])


def complete_graph(N: int) -> np.ndarray:
    """All-reduce: every node receives from every node."""
    return np.tile(np.arange(N, dtype=np.int64), (N, 1))


def identity_graph(N: int) -> np.ndarray:
    """k = 0: no communication (each worker keeps its own model)."""
    return np.arange(N, dtype=np.int64).reshape(N, 1)


def _admissible_permutation(rng: SplitMix64, in_nbrs):
    """One Fisher-Yates draw; None as soon as a finalised slot t holds t
    itself or an existing in-neighbour of t."""
    n = len(in_nbrs)
    sigma = list(range(n))
    for t in range(n - 1, 0, -1):
        j = rng.uniform(t + 1)
        sigma[t], sigma[j] = sigma[j], sigma[t]
        if sigma[t] == t or sigma[t] in in_nbrs[t]:
            return None
    if sigma[0] == 0 or sigma[0] in in_nbrs[0]:
        return None
    return sigma


def random_regular_graph(N: int, k: int, graph_seed: int, rnd: int = 0) -> np.ndarray:
    """Seeded random k-regular directed graph (self-loops added), see module
    docstring for the exact construction."""
    if not (1 <= k <= N - 1):
        raise GraphError("random regular graph needs 1 <= k <= N-1")
    rng = SplitMix64(round_state(graph_seed, rnd))
    pi = fisher_yates(rng, N)
    in_nbrs = [set() for _ in range(N)]
    for t in range(N):
        in_nbrs[pi[(t + 1) % N]].add(pi[t])
    for _layer in range(k - 1):
        for _try in range(MAX_LAYER_TRIES):
            sigma = _admissible_permutation(rng, in_nbrs)
            if sigma is not None:
                for i in range(N):
                    in_nbrs[i].add(sigma[i])
                break
        else:
            raise GraphError("no admissible permutation layer after %d draws" % MAX_LAYER_TRIES)
    return _rows_from_in_neighbours(in_nbrs)


def build_graph(kind: str, N: int, k: int, graph_seed: int = 0, rnd: int = 0):
    """Return (nbr, wgt): nbr [N, k+1] ascending with self included, wgt the
    equal weights 1/(k+1) (fp64)."""
    if kind == "ring":
        nbr = ring_graph(N)
    elif kind == "root":
        nbr = root_graph(N)
    elif kind == "complete":
        nbr = complete_graph(N)
    elif kind == "identity":
        nbr = identity_graph(N)
    elif kind == "random_regular":
        nbr = random_regular_graph(N, k, graph_seed, rnd)
    else:
        raise GraphError("unknown graph kind %r" % kind)
    if nbr.shape[1] != k + 1:
        raise GraphError("kind %r gives %d neighbours per row, not k+1=%d" % (kind, nbr.shape[1], k + 1))
    wgt = np.full(nbr.shape, 1.0 / nbr.shape[1])
    return nbr, wgt


def default_kind(N: int, k: int) -> str:
    if k == 0:
        return "identity"
    if k == N - 1:
        return "complete"
    if k == 1:
        return "ring"
    return "random_regular"


def mixing_matrix(nbr: np.ndarray, wgt: np.ndarray) -> np.ndarray:
    """Dense P with P[i, nbr[i, m]] = wgt[i, m] (Appendix A)."""
    N = nbr.shape[0]
    P = np.zeros((N, N))
    for i in range(N):
        for m in range(nbr.shape[1]):
            P[i, nbr[i, m]] += wgt[i, m]
    return P


def adjacency_mixing(A: np.ndarray) -> np.ndarray:
    """P = diag(d_in)^-1 A for a 0/1 adjacency with self-loops, rows = receivers."""
    A = np.asarray(A, dtype=np.float64)
    return A / A.sum(axis=1, keepdims=True)


def spectral_gap(P: np.ndarray) -> float:
    """1 - sigma_2(P), sigma_2 the second largest singular value (Appendix A)."""
    s = np.linalg.svd(P, compute_uv=False)
    return float(1.0 - s[1]) if s.shape[0] > 1 else 1.0


def is_doubly_stochastic(P: np.ndarray, tol: float = 1e-12) -> bool:
    return bool(np.all(np.abs(P.sum(axis=0) - 1) <= tol) and np.all(np.abs(P.sum(axis=1) - 1) <= tol)
                and np.all(P >= 0))
