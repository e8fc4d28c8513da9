"""GB300-native MixFP4 W4A4 linear layer (arXiv 2605.31035).

The compute path is hand-written CUDA for sm_103a behind the C-ABI library
``libmixfp4.so`` (declared in ``include/mixfp4.h``); ``ops`` is a thin ctypes
binding with the same entry-point names.  The binding is loaded lazily so that
the input generators in ``synth`` import without a GPU; any compute call
without the built library raises instead of falling back.
"""
from __future__ import annotations

__all__ = ["ops", "synth"]


def __getattr__(name):
    if name in __all__:
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
