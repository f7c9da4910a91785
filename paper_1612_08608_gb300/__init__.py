"""GB300-native data-parallel hot path of ASAP (Kadav & Kruus, arXiv
1612.08608): N simulated workers on one GPU, each taking a minibatch SGD
step on its own shard, followed by the stochastic reduce W <- P W over a
sparse doubly-stochastic mixing graph, with NOTIFY-ACK kept as per-worker
round counters.  The compute path is libasap.so (CUDA, sm_103a) behind the
C ABI in include/asap.h; this package only marshals arguments.

``inputs`` (seeded synthetic data) imports without the CUDA library;
``Context`` and ``build_graph`` load it on first use.
"""
__all__ = ["Context", "AsapError", "build_graph", "load_library", "inputs"]


def __getattr__(name):
    if name in ("Context", "AsapError", "build_graph"):
        from . import api
        return getattr(api, name)
    if name == "load_library":
        from ._lib import load_library
        return load_library
    raise AttributeError(name)
