"""DeltaS hot path on GB300: gated-delta-rule chunk update with fused state drift, chunk
scoring, retain selection and in-place KV compaction, as CUDA kernels behind a C ABI
(``include/deltas.h``).

The Python functions exported here are a thin ctypes binding (argument marshalling only); every
step runs in the library's kernels.  The binding is loaded lazily so that the input generators
and configs can be imported without the compiled library.
"""
from __future__ import annotations

__all__ = ["lib"]


def __getattr__(name):
    if name == "lib":
        from . import _lib
        return _lib
    raise AttributeError(name)
