"""Python binding of the ASAP C ABI (include/asap.h): argument marshalling
only.  Every step of a round runs in the CUDA kernels of libasap.so."""
from __future__ import annotations

import ctypes as C
from typing import Optional, Sequence

import numpy as np

from ._lib import load_library

STATUS = {0: "ASAP_OK", 1: "ASAP_ERR_ARG", 2: "ASAP_ERR_CUDA", 3: "ASAP_ERR_OOM",
          4: "ASAP_ERR_TIMEOUT", 5: "ASAP_ERR_STATE", 6: "ASAP_ERR_GRAPH"}
GRAPH = {"ring": 1, "root": 2, "random_regular": 3, "complete": 4, "explicit": 5, "identity": 6}
LOSS = {"none": 0, "hinge": 1, "logistic": 2, "softmax": 3}
RESIDENCY = {"device": 0, "host": 1}
LR_SCHEDULE = {"constant": 0, "inverse": 1}
SYNC = {"bsp": 0, "notify_ack": 1, "async": 2}


class AsapError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__("%s: %s" % (STATUS.get(status, status), message))
        self.status = status
        self.name = STATUS.get(status, str(status))


def _check(lib, ctx, status: int):
    if status != 0:
        msg = lib.asap_last_error(ctx)
        raise AsapError(status, msg.decode() if msg else "")


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _ptr_array(arrs):
    return (C.c_void_p * len(arrs))(*[None if a is None else _ptr(a) for a in arrs])


def build_graph(kind: str, N: int, k: int, graph_seed: int = 0, rnd: int = 0) -> np.ndarray:
    """Host graph builder of the library (no GPU needed): [N, k+1] int32."""
    lib = load_library()
    out = np.empty((N, k + 1), dtype=np.int32)
    _check(lib, None, lib.asap_build_graph(GRAPH[kind], N, k, graph_seed, rnd, _ptr(out)))
    return out


def debug_batch_image(shards, batch: int, slab_cols: int, t: int, ctas_per_worker: int = 1):
    """The image asap_load_shards builds for minibatch t (host only, for
    tests): (image bytes uint8, desc [N, 8] int64, (list byte offset, slab
    offsets byte offset, list length))."""
    lib = load_library()
    rp = [np.ascontiguousarray(a, dtype=np.int64) for a in shards.rowptr]
    cl = [np.ascontiguousarray(a, dtype=np.int32) for a in shards.col]
    vl = [np.ascontiguousarray(a, dtype=np.float32) for a in shards.val]
    yl = [np.ascontiguousarray(a, dtype=np.float32) for a in shards.y]
    N = len(rp)
    if t < 0 or any((t + 1) * batch > a.shape[0] - 1 for a in rp):
        raise ValueError("minibatch %d of %d rows is past the end of a shard" % (t, batch))
    args = (N, shards.d, batch, slab_cols, ctas_per_worker, t, _ptr_array(rp), _ptr_array(cl), _ptr_array(vl),
            _ptr_array(yl))
    size = C.c_int64()
    desc = np.empty((N, 8), dtype=np.int64)
    lst = np.empty(3, dtype=np.int64)
    st = lib.asap_debug_batch_image(*args, None, 0, C.byref(size), _ptr(desc), _ptr(lst))
    if st != 1:                       # anything but "buffer too small" is a real error
        _check(lib, None, st)
    img = np.empty(size.value, dtype=np.uint8)
    _check(lib, None, lib.asap_debug_batch_image(*args, _ptr(img), img.shape[0], C.byref(size), _ptr(desc),
                                                 _ptr(lst)))
    return img, desc, (int(lst[0]), int(lst[1]), int(lst[2]))


class Context:
    """N simulated workers on the current CUDA device (see include/asap.h)."""

    row_dtype = np.float32   # parameter rows as read_rows returns them

    def __init__(self, N: int, d: int, graph_seed: int = 0, k: int = 0):
        self._lib = load_library()
        h = C.c_void_p()
        _check(self._lib, None, self._lib.asap_create(N, d, graph_seed, k, C.byref(h)))
        self._h = h
        self.N, self.d, self.k = N, d, k
        self.P = d
        self._keep = []

    # -- configuration -------------------------------------------------
    def _c(self, status):
        _check(self._lib, self._h, status)

    def set_graph(self, kind: str, regenerate: bool = False):
        self._c(self._lib.asap_set_graph(self._h, GRAPH[kind], int(regenerate)))

    def set_mixing(self, nbr, wgt):
        nbr = np.ascontiguousarray(nbr, dtype=np.int32)
        wgt = np.ascontiguousarray(wgt, dtype=np.float32)
        self._c(self._lib.asap_set_mixing(self._h, _ptr(nbr), _ptr(wgt)))

    def set_model(self, loss: str, batch: int, lr: float, num_classes: int = 1, l2: float = 0.0):
        self._c(self._lib.asap_set_model(self._h, LOSS[loss], num_classes, batch, lr, l2))
        self.P = self.d * (num_classes if loss == "softmax" else 1)

    def set_schedule(self, local_steps: int = 1, lr_schedule: str = "constant", gamma: float = 0.0):
        """local_steps minibatch steps per worker per round; learning rate
        ``constant`` (eta_k = lr) or ``inverse`` (eta_k = lr / (1 + gamma k)),
        k = round * local_steps + step."""
        self._c(self._lib.asap_set_schedule(self._h, int(local_steps), LR_SCHEDULE[lr_schedule], float(gamma)))

    def set_stream(self, stream):
        """stream: a torch.cuda.Stream, an integer cudaStream_t, or None."""
        handle = getattr(stream, "cuda_stream", stream)
        self._c(self._lib.asap_set_stream(self._h, C.c_void_p(handle) if handle else None))

    def set_shard_residency(self, where: str):
        self._c(self._lib.asap_set_shard_residency(self._h, RESIDENCY[where]))

    def shard_block_bytes(self, rnd: int) -> int:
        v = C.c_uint64()
        self._c(self._lib.asap_shard_block_bytes(self._h, rnd, C.byref(v)))
        return v.value

    def load_shards(self, shards=None, rowptr=None, col=None, val=None, y=None):
        if shards is not None:
            rowptr, col, val, y = shards.rowptr, shards.col, shards.val, shards.y
        # None: a worker that a worker-sharded context does not step
        def conv(arrs, dt):
            return [None if a is None else np.ascontiguousarray(a, dtype=dt) for a in arrs]
        rp, cl, vl, yl = conv(rowptr, np.int64), conv(col, np.int32), conv(val, np.float32), conv(y, np.float32)
        n = np.array([0 if a is None else a.shape[0] - 1 for a in rp], dtype=np.int64)
        self._c(self._lib.asap_load_shards(self._h, _ptr_array(rp), _ptr_array(cl), _ptr_array(vl),
                                           _ptr_array(yl), _ptr(n)))

    def load_dense_shards(self, shards=None, X=None, y=None):
        if shards is not None:
            X, y = shards.X, shards.y
        xl = [np.ascontiguousarray(a, dtype=np.uint16) for a in X]
        yl = [np.ascontiguousarray(a, dtype=np.int32) for a in y]
        n = np.array([a.shape[0] for a in xl], dtype=np.int64)
        self._c(self._lib.asap_load_dense_shards(self._h, _ptr_array(xl), _ptr_array(yl), _ptr(n)))

    # -- the round -----------------------------------------------------
    def local_step(self):
        self._c(self._lib.asap_local_step(self._h))

    def stochastic_reduce(self):
        self._c(self._lib.asap_stochastic_reduce(self._h))

    def round(self, T: int = 1):
        self._c(self._lib.asap_round(self._h, T))

    def sync(self):
        self._c(self._lib.asap_sync(self._h))

    # -- state ---------------------------------------------------------
    def read_params(self, out: Optional[np.ndarray] = None):
        if out is None:
            out = np.empty((self.N, self.P), dtype=np.float32)
        r = C.c_int64()
        self._c(self._lib.asap_read_params(self._h, _ptr(out), C.byref(r)))
        return out, r.value

    def write_params(self, W: np.ndarray, rnd: int = 0):
        W = np.ascontiguousarray(W, dtype=np.float32)
        assert W.shape == (self.N, self.P)
        self._c(self._lib.asap_write_params(self._h, _ptr(W), rnd))

    def write_params_device(self, W, rnd: int = 0):
        """W: a CUDA tensor (float32, N x P with unit column stride) on the
        context's device; copied device to device."""
        assert W.dtype.itemsize == 4 and W.dim() == 2 and W.shape[0] == self.N and W.shape[1] >= self.P
        assert W.stride(1) == 1 and W.is_cuda
        self._c(self._lib.asap_write_params_device(self._h, C.c_void_p(W.data_ptr()), W.stride(0), rnd))

    def read_param_columns(self, first: int, count: int, out: Optional[np.ndarray] = None):
        """Columns [first, first + count) of every worker's parameters."""
        if out is None:
            out = np.empty((self.N, count), dtype=np.float32)
        self._c(self._lib.asap_read_param_columns(self._h, first, count, _ptr(out)))
        return out

    def read_metrics(self, first: int, count: int):
        loss = np.empty(count, dtype=np.float32)
        cons = np.empty(count, dtype=np.float32)
        self._c(self._lib.asap_read_metrics(self._h, first, count, _ptr(loss), _ptr(cons)))
        return loss, cons

    def read_counters(self):
        a, b, c = C.c_uint64(), C.c_uint64(), C.c_uint64()
        self._c(self._lib.asap_read_counters(self._h, C.byref(a), C.byref(b), C.byref(c)))
        return {"reduces": a.value, "consistent_inputs": b.value, "timeouts": c.value}

    def get_graph(self, rnd: int = 0):
        nbr = np.empty((self.N, self.k + 1), dtype=np.int32)
        wgt = np.empty((self.N, self.k + 1), dtype=np.float32)
        self._c(self._lib.asap_get_graph(self._h, rnd, _ptr(nbr), _ptr(wgt)))
        return nbr, wgt

    def set_sync_mode(self, mode: str):
        """``bsp``, ``notify_ack`` or ``async`` (measurement only)."""
        self._c(self._lib.asap_set_sync_mode(self._h, SYNC[mode]))

    def set_worker_order(self, order=None):
        """Cluster q of the local step runs worker order[q] (None: identity)."""
        if order is None:
            self._c(self._lib.asap_set_worker_order(self._h, None))
            return
        order = np.ascontiguousarray(order, dtype=np.int32)
        self._c(self._lib.asap_set_worker_order(self._h, _ptr(order)))

    # -- worker-sharded mode ---------------------------------------------
    def set_worker_range(self, first: int, count: int):
        """Step only workers [first, first + count); the others' rows are
        delivered with write_rows every round."""
        self._c(self._lib.asap_set_worker_range(self._h, first, count))

    def read_rows(self, rows, out: Optional[np.ndarray] = None):
        """Rows of W_t as stored, and the factor that gives their true values."""
        rows = np.ascontiguousarray(rows, dtype=np.int32)
        if out is None:
            out = np.empty((rows.shape[0], self.P), dtype=np.float32)
        sc = C.c_float()
        self._c(self._lib.asap_read_rows(self._h, _ptr(rows), rows.shape[0], _ptr(out), C.byref(sc)))
        return out, sc.value

    def write_rows(self, rows, values: np.ndarray):
        rows = np.ascontiguousarray(rows, dtype=np.int32)
        values = np.ascontiguousarray(values, dtype=np.float32)
        assert values.shape == (rows.shape[0], self.P)
        self._c(self._lib.asap_write_rows(self._h, _ptr(rows), rows.shape[0], _ptr(values)))

    def read_consistency(self):
        """{inputs_read, inputs_current} of the gated reduces since creation."""
        a, b = C.c_uint64(), C.c_uint64()
        self._c(self._lib.asap_read_consistency(self._h, C.byref(a), C.byref(b)))
        return {"inputs_read": a.value, "inputs_current": b.value}

    def set_wait_limit_ns(self, ns: int):
        self._c(self._lib.asap_set_wait_limit_ns(self._h, ns))

    def debug_skip_notify(self, worker: int):
        self._c(self._lib.asap_debug_skip_notify(self._h, worker))

    KERNELS = ("local_step", "reduce", "dense_fwd", "dense_grad", "apply", "gather")

    def set_kernel_timing(self, enable: bool = True):
        self._c(self._lib.asap_set_kernel_timing(self._h, int(enable)))

    def read_kernel_times(self):
        """{kernel: (timed launches, total ms)} since enabling / the last read."""
        n = np.zeros(len(self.KERNELS), dtype=np.uint64)
        ms = np.zeros(len(self.KERNELS), dtype=np.float64)
        self._c(self._lib.asap_read_kernel_times(self._h, _ptr(n), _ptr(ms)))
        return {k: (int(n[i]), float(ms[i])) for i, k in enumerate(self.KERNELS)}

    def kernel_launches(self) -> int:
        v = C.c_uint64()
        self._c(self._lib.asap_kernel_launches(self._h, C.byref(v)))
        return v.value

    def close(self):
        if getattr(self, "_h", None):
            self._lib.asap_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
