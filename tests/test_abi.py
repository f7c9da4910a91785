"""The C ABI library builds, loads and exports every symbol include/asap.h
declares; its host graph builder matches the oracle bit for bit.  No GPU."""
import os
import re

import numpy as np
import pytest

from oracle import graphs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_1612_08608_gb300 import build
    build.build()
    from paper_1612_08608_gb300._lib import load_library
    return load_library()


def _header_functions():
    text = open(os.path.join(ROOT, "include", "asap.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(asap_[a-z_0-9]+)\s*\(", text)))


def test_header_symbols_exported(lib):
    from paper_1612_08608_gb300._lib import SIGNATURES
    names = _header_functions()
    assert len(names) >= 20
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(SIGNATURES), set(names) ^ set(SIGNATURES)
    assert lib.asap_version().startswith(b"asap-gb300")


@pytest.mark.parametrize("kind,N,k", [("ring", 2, 1), ("ring", 33, 1), ("root", 4, 2), ("root", 25, 2),
                                      ("root", 256, 2), ("complete", 7, 6), ("identity", 3, 0),
                                      ("random_regular", 16, 2), ("random_regular", 64, 4),
                                      ("random_regular", 256, 4), ("random_regular", 5, 3),
                                      ("random_regular", 100, 7), ("random_regular", 2, 1)])
def test_graph_builder_bit_exact_with_oracle(lib, kind, N, k):
    from paper_1612_08608_gb300 import build_graph
    for seed in (0, 1, 2 ** 63 + 5):
        for rnd in (0, 1, 7, 1000):
            got = build_graph(kind, N, k, graph_seed=seed, rnd=rnd)
            want, _ = graphs.build_graph(kind, N, k, seed, rnd)
            assert np.array_equal(got, want), (kind, N, k, seed, rnd)


def test_graph_builder_rejects_bad_kinds(lib):
    from paper_1612_08608_gb300 import AsapError, build_graph
    for kind, N, k in [("ring", 4, 2), ("root", 3, 2), ("complete", 5, 3), ("random_regular", 4, 0)]:
        with pytest.raises(AsapError):
            build_graph(kind, N, k)


def test_create_rejects_bad_sizes_and_reports_a_missing_device(lib):
    import ctypes as C
    h = C.c_void_p()
    for N, d, k in [(0, 10, 0), (4, 0, 1), (4, 10, 4), (4, 10, -1), (2000, 10, 1), (64, 10, 40)]:
        assert lib.asap_create(N, d, 0, k, C.byref(h)) == 1, (N, d, k)   # ASAP_ERR_ARG
        assert not h.value
        assert lib.asap_last_error(None)
    import torch
    if torch.cuda.is_available():
        pytest.skip("a device is present")
    # No device: the context's first CUDA call fails; nothing is returned.
    assert lib.asap_create(4, 10, 0, 1, C.byref(h)) == 2                  # ASAP_ERR_CUDA
    assert not h.value
    assert lib.asap_last_error(None)
