"""asap_mix_noalloc, the entry point for callers that cannot allocate device
memory (a framework that owns all of HBM through its own pool, or a
latency-critical loop where cudaMalloc may synchronise the device).

It is called here through the C ABI on buffers the test owns, and its output
is checked against the context's own stochastic reduce and against the CPU
oracle (Eq. A.1, second line, and the consensus error) on two calls in a
row (the second call starts from the first call's output, so the shared
scratch array holds the previous call's contents).  After a warm-up call,
further calls do not lower the device's free memory and leave torch's
allocation count unchanged.  Collected last on purpose: a run that stops at the first
failure has already run every other test."""
import ctypes as C
import gc

import numpy as np
import pytest

from oracle import reduce
from paper_1612_08608_gb300 import inputs
from parity import rel_err_rows

pytestmark = pytest.mark.gpu


def _noalloc(lib, W_in, W_out, N, d, ld, nbr, wgt, kp1, cons, stream):
    return lib.asap_mix_noalloc(C.c_void_p(W_in.data_ptr()), C.c_void_p(W_out.data_ptr()), N, d, ld,
                                C.c_void_p(nbr.data_ptr()), C.c_void_p(wgt.data_ptr()), kp1,
                                C.c_void_p(cons.data_ptr()), C.c_void_p(stream))


@pytest.mark.parametrize("N,d,k", [(32, 100003, 2), (8, 4093, 1), (256, 20000, 4)])
def test_mix_noalloc_matches_stochastic_reduce_twice(N, d, k):
    import torch

    from paper_1612_08608_gb300 import Context
    from paper_1612_08608_gb300._lib import load_library

    lib = load_library()
    W0 = inputs.mixing_params(seed=3, N=N, d=d)
    kind = "ring" if k == 1 else "random_regular"
    with Context(N, d, graph_seed=1, k=k) as ctx:
        ctx.set_graph(kind)
        ctx.write_params(W0, 0)
        ref_W, ref_c = [], []
        for t in range(2):
            ctx.stochastic_reduce()
            ref_W.append(ctx.read_params()[0])
            ref_c.append(float(ctx.read_metrics(t, 1)[1][0]))
        nbr, wgt = ctx.get_graph(0)

    ld = (d + 3) // 4 * 4
    dev = torch.device("cuda", torch.cuda.current_device())
    W_a = torch.zeros(N, ld, dtype=torch.float32, device=dev)
    W_a[:, :d] = torch.from_numpy(W0).to(dev)
    W_b = torch.empty_like(W_a)
    cons = torch.empty(1, dtype=torch.float32, device=dev)
    d_nbr = torch.from_numpy(nbr).to(dev)
    d_wgt = torch.from_numpy(wgt).to(dev)
    stream = torch.cuda.current_stream().cuda_stream
    prev = W0.astype(np.float64)
    for t in range(2):
        src, dst = (W_a, W_b) if t == 0 else (W_b, W_a)
        assert _noalloc(lib, src, dst, N, d, ld, d_nbr, d_wgt, k + 1, cons, stream) == 0, \
            lib.asap_last_error(None)
        torch.cuda.synchronize()
        got = dst[:, :d].cpu().numpy()
        assert rel_err_rows(got, ref_W[t]) <= 1e-5, t
        assert abs(cons.item() - ref_c[t]) <= 1e-4 * ref_c[t] + 1e-6, (t, cons.item(), ref_c[t])
        assert torch.all(dst[:, d:] == 0)   # zero padding columns stay zero
        # the oracle, restarted from this call's input
        want = reduce.stochastic_reduce(prev, nbr.astype(np.int64), wgt.astype(np.float64))
        assert rel_err_rows(got, want) <= 1e-5, t
        cw = reduce.consensus_error(want)
        assert abs(cons.item() - cw) <= 1e-4 * cw + 1e-6, (t, cons.item(), cw)
        prev = got.astype(np.float64)

    # No allocation: free device memory does not drop and torch's count stays
    # put.  Contexts of earlier tests are collected first; one released while
    # the calls run could only raise the free figure, never lower it.
    gc.collect()
    torch.cuda.synchronize()
    free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
    for t in range(6):
        src, dst = (W_a, W_b) if t % 2 == 0 else (W_b, W_a)
        assert _noalloc(lib, src, dst, N, d, ld, d_nbr, d_wgt, k + 1, cons, stream) == 0
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] >= free0
    assert torch.cuda.memory_allocated() == alloc0


def test_mix_noalloc_rejects_sizes_beyond_its_scratch():
    import torch

    from paper_1612_08608_gb300._lib import load_library
    lib = load_library()
    dev = torch.device("cuda", torch.cuda.current_device())
    x = torch.zeros(4, dtype=torch.float32, device=dev)
    n = torch.zeros(4, dtype=torch.int32, device=dev)
    ld_too_big = 256 * 16 * 32768 + 4            # N = 256 allows 524,288 columns
    assert _noalloc(lib, x, x.clone(), 256, ld_too_big, ld_too_big, n, x, 1, x, 0) == 1
    assert b"scratch" in lib.asap_last_error(None)
    assert _noalloc(lib, x, x.clone(), 257, 4, 4, n, x, 1, x, 0) == 1
    # overlapping input and output ranges (not only equal base pointers)
    big = torch.zeros(4 * 16 + 8, dtype=torch.float32, device=dev)
    assert _noalloc(lib, big[8:], big[:64], 4, 16, 16, n, x, 1, x, 0) == 1
    assert b"overlap" in lib.asap_last_error(None)
