"""GB300-native HyperDFlash block-drafting path.

The compute lives in ``libhdf.so`` (hand-written CUDA for sm_103a behind a
C ABI, see ``include/hdf.h``); ``paper_2606_26744_gb300.hdf`` is the thin
ctypes binding and ``paper_2606_26744_gb300.workloads`` draws seeded inputs.
Importing the package itself loads nothing.
"""
__all__ = ["hdf", "workloads"]
