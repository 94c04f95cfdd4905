"""BRISK-DLM decode tail on GB300 (sm_103a).

The compute runs in the CUDA library built from ``csrc/``; ``brisk`` is its
thin ctypes binding (loaded on first use); ``loop`` drives captured tails block after
block with double-buffered inputs. ``synth`` builds seeded synthetic inputs shaped like the
paper's workloads.
"""
import importlib

__all__ = ["synth", "brisk", "build", "loop"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
