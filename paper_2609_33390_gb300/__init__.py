"""BRISK-DLM decode tail on GB300 (sm_103a).

The compute runs in the CUDA library built from ``csrc/``; ``brisk`` is its
thin ctypes binding (loaded on first use). ``synth`` builds seeded synthetic
inputs shaped like the paper's workloads.
"""
__all__ = ["synth", "brisk"]


def __getattr__(name):
    if name == "brisk":
        from . import brisk as _b
        return _b
    if name == "synth":
        from . import synth as _s
        return _s
    raise AttributeError(name)
