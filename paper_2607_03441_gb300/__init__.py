"""GB300-native (sm_103a) hot path of the aTTT in-episode update step.

The compute lives in ``libattt.so`` (hand-written CUDA under ``csrc/``), whose
C ABI is declared in ``include/attt.h``.  ``paper_2607_03441_gb300.attt`` is a
thin ctypes binding with the same names; ``workloads`` draws the seeded
synthetic inputs.  Importing this package loads nothing: the library is
loaded on first use of the binding and fails loudly if it is missing.
"""
__all__ = ["attt", "workloads", "build"]
