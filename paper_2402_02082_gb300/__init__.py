"""GliDe-with-CaPE KV-cache attention hot path for GB300 (sm_103a).

The compute lives in ``libglide.so`` (hand-written CUDA kernels behind a C ABI
declared in ``include/glide.h``); ``binding`` marshals torch tensors into that
ABI.  ``synth`` draws seeded synthetic inputs.  Importing the package does not
load the library; the first binding call does, and fails loudly if it has not
been built.
"""
import importlib

__all__ = ["binding", "synth"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
