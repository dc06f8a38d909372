"""GB300-native batched statevector engine for static parametrised circuits.

The compute path is the C-ABI library ``libvqc.so`` (host compiler + sm_103a
kernels, sources under ``csrc/``); ``binding`` is a thin ctypes layer with the
same entry-point names, and ``circuit`` wraps it for PyTorch tensors and
autograd.  Submodules load lazily so that the seeded input generators
(``workloads``) import without a GPU or a built library.
"""
import importlib

__all__ = ["binding", "circuit", "workloads"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module("." + name, __name__)
    if name in ("Circuit", "VQCFunction"):
        return getattr(importlib.import_module(".circuit", __name__), name)
    raise AttributeError(name)
