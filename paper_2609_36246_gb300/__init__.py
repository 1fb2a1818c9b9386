"""GB300 (sm_103a) implementation of the OLIVE per-token scoring path.

The compute lives in ``libolive.so`` (hand-written CUDA for sm_103a behind a
C ABI, declared in ``include/olive.h``); :mod:`.binding` is a thin ctypes
layer over it with the same entry-point names, and :mod:`.synth` draws the
seeded synthetic workloads.  Importing the package loads nothing: the library
is opened on first use and a missing or unbuildable library raises.
"""

__all__ = ["binding", "synth", "build"]
