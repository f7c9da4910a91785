"""ctypes loader for libasap.so, the only compute path of this package.

There is no CPU fallback: if the library is missing or does not load, every
call raises.  Build it with ``paper_1612_08608_gb300.build.build()`` (or
``__graft_entry__.build()``).
"""
from __future__ import annotations

import ctypes as C
import os

_LIB = None
LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libasap.so")

# Every symbol include/asap.h declares, with its (restype, argtypes).
_P = C.c_void_p
SIGNATURES = {
    "asap_create": (C.c_int, [C.c_int, C.c_int64, C.c_uint64, C.c_int, C.POINTER(_P)]),
    "asap_set_graph": (C.c_int, [_P, C.c_int, C.c_int]),
    "asap_set_mixing": (C.c_int, [_P, _P, _P]),
    "asap_set_model": (C.c_int, [_P, C.c_int, C.c_int, C.c_int, C.c_float, C.c_float]),
    "asap_set_schedule": (C.c_int, [_P, C.c_int, C.c_int, C.c_float]),
    "asap_debug_batch_image": (C.c_int, [C.c_int, C.c_int64, C.c_int, C.c_int, C.c_int, C.c_int, _P, _P, _P, _P, _P,
                                         C.c_int64, _P, _P, _P]),
    "asap_set_stream": (C.c_int, [_P, _P]),
    "asap_set_shard_residency": (C.c_int, [_P, C.c_int]),
    "asap_shard_block_bytes": (C.c_int, [_P, C.c_int64, C.POINTER(C.c_uint64)]),
    "asap_load_shards": (C.c_int, [_P, _P, _P, _P, _P, _P]),
    "asap_load_dense_shards": (C.c_int, [_P, _P, _P, _P]),
    "asap_local_step": (C.c_int, [_P]),
    "asap_stochastic_reduce": (C.c_int, [_P]),
    "asap_round": (C.c_int, [_P, C.c_int]),
    "asap_sync": (C.c_int, [_P]),
    "asap_read_params": (C.c_int, [_P, _P, C.POINTER(C.c_int64)]),
    "asap_write_params": (C.c_int, [_P, _P, C.c_int64]),
    "asap_write_params_device": (C.c_int, [_P, _P, C.c_int64, C.c_int64]),
    "asap_read_param_columns": (C.c_int, [_P, C.c_int64, C.c_int64, _P]),
    "asap_read_metrics": (C.c_int, [_P, C.c_int64, C.c_int64, _P, _P]),
    "asap_read_counters": (C.c_int, [_P, C.POINTER(C.c_uint64), C.POINTER(C.c_uint64), C.POINTER(C.c_uint64)]),
    "asap_get_graph": (C.c_int, [_P, C.c_int64, _P, _P]),
    "asap_set_wait_limit_ns": (C.c_int, [_P, C.c_uint64]),
    "asap_set_sync_mode": (C.c_int, [_P, C.c_int]),
    "asap_set_worker_order": (C.c_int, [_P, _P]),
    "asap_set_worker_range": (C.c_int, [_P, C.c_int, C.c_int]),
    "asap_read_rows": (C.c_int, [_P, _P, C.c_int, _P, C.POINTER(C.c_float)]),
    "asap_write_rows": (C.c_int, [_P, _P, C.c_int, _P]),
    "asap_read_consistency": (C.c_int, [_P, C.POINTER(C.c_uint64), C.POINTER(C.c_uint64)]),
    "asap_debug_skip_notify": (C.c_int, [_P, C.c_int]),
    "asap_set_kernel_timing": (C.c_int, [_P, C.c_int]),
    "asap_read_kernel_times": (C.c_int, [_P, _P, _P]),
    "asap_kernel_launches": (C.c_int, [_P, C.POINTER(C.c_uint64)]),
    "asap_build_graph": (C.c_int, [C.c_int, C.c_int, C.c_int, C.c_uint64, C.c_int64, _P]),
    "asap_mix_noalloc": (C.c_int, [_P, _P, C.c_int, C.c_int64, C.c_int64, _P, _P, C.c_int, _P, _P]),
    "asap_last_error": (C.c_char_p, [_P]),
    "asap_version": (C.c_char_p, []),
    "asap_destroy": (None, [_P]),
}


def load_library(path: str = LIB_PATH) -> C.CDLL:
    """Load (once) and type the C ABI.  Raises if the library is absent."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(path):
        raise RuntimeError("libasap.so not found at %s: build it first (paper_1612_08608_gb300.build)" % path)
    lib = C.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = lib
    return lib
