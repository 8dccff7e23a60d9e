"""GB300-native branch-decode step for Hierarchical Parallel Decoding.

The compute lives in ``libhpd.so`` (hand-written CUDA for sm_103a behind a C
ABI, declared in ``include/hpd.h``).  ``hpd`` is the thin ctypes binding with
the same entry-point names; ``workloads`` draws seeded synthetic inputs.
Importing the package loads nothing; the library is loaded on first use and
a missing library is an error, never a fallback.
"""

__all__ = ["hpd", "workloads"]
