"""GB300-native what-if placement simulation (SliceScheduler's Global Simulator).

The hot path lives in ``libgmgsim.so`` (hand-written sm_103a CUDA behind the C
ABI of ``include/gmgsim.h``); ``gmgsim`` is the thin ctypes binding and
``workloads`` generates the seeded synthetic inputs.
"""
from . import workloads  # noqa: F401
