"""CPU oracle for ASAP's data-parallel hot path (arXiv 1612.08608).

TEST INFRASTRUCTURE ONLY.  This package is the slow, plain, fp64 statement
of what one ASAP round computes; it exists so that the CUDA path can be
checked against it.  Only the test suite, ``__graft_entry__.smoke()`` and
the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import
it.  The library itself never calls it and has no CPU fallback.

It shares no code with the CUDA path: no headers, kernels, constants, table
generators or pre/post-processing.  Inputs come from
``paper_1612_08608_gb300.inputs`` (data draws only) and from explicit arrays.

Modules
-------
graphs   -- Section 3.1 / Fig. 2 / Appendix A: communication graphs, the
            mixing matrix P = diag(d_in)^-1 A, the spectral gap 1 - sigma_2(P),
            and the seeded generator that builds a graph per round.
sgd      -- Eq. A.1 first line: one minibatch SGD step per worker (hinge,
            logistic, and the bf16-input softmax-regression variant).
reduce   -- Eq. A.1 second line: the stochastic reduce W <- P W, plus the
            consensus error ||W - 1 wbar^T||_F.
rounds   -- Eq. A.1 iterated: SGD step then stochastic reduce, per round.

Parity status: every function here is pinned by a ``-m "not gpu"`` test in
``tests/test_oracle_*.py`` except the paper's printed spectral gaps for its
"expander" (0.38 / 0.2) and parameter-server (0.75 / 0.68) drawings in
Fig. 2, which no graph convention reproduces: those two numbers are parity
unpinned (the graph builder itself is pinned by closed forms instead).
"""
