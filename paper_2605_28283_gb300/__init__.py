"""GB300-native PrunePath sparse-FFN path.

The compute lives in ``libprunepath.so`` (hand-written CUDA for sm_103a behind
the C ABI declared in ``include/prunepath.h``).  ``binding`` is a thin ctypes
layer over it with the same entry-point names; ``workloads`` holds the seeded
synthetic-input recipes.  Importing this package does not load the CUDA
library: the first call into ``binding`` does, and raises if it is missing.
"""

__all__ = ["binding", "workloads"]
