"""Brute-force optimal CPU/GPU device-mapping search on GB300 (sm_103a).

The search runs in hand-written CUDA kernels behind the C ABI declared in
``include/bf.h`` (``libbf.so``); :mod:`paper_2607_22242_gb300.bf` is the thin
ctypes binding and :mod:`paper_2607_22242_gb300.scenarios` the seeded input
generator.  Importing this package loads nothing; the binding loads the library
on first use and raises if it is missing.
"""
__all__ = ["bf", "scenarios"]
