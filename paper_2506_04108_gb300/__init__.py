"""GB300-native (sm_103a) decode-time attention path of Rectified Sparse Attention.

The compute lives in ``libresa.so`` (hand-written CUDA, C ABI declared in
``include/resa.h``); :mod:`paper_2506_04108_gb300.resa` is the thin ctypes
binding. :mod:`paper_2506_04108_gb300.synth` draws seeded synthetic inputs.
Importing the package does not load the library; the binding loads it on
first use and raises if it has not been built.
"""
__all__ = ["resa", "synth"]
