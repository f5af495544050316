"""GB300-native DAVET step-conditioning hot path.

The compute path lives in the CUDA library ``libdavet.so`` (sources in
``csrc/``, C ABI declared in ``include/davet.h``).  ``load()`` returns the
thin ctypes binding; it raises if the library is missing or cannot load:
there is no CPU fallback.
"""
from __future__ import annotations

__all__ = ["load", "build"]


def build(verbose: bool = False) -> str:
    from . import _build
    return _build.build(verbose=verbose)


def load():
    from . import davet
    return davet.load()
