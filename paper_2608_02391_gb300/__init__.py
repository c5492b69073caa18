"""GB300-native CoPES evolution-strategy core.

The compute lives in the CUDA library ``libcopes.so`` (built from ``csrc/`` for sm_103a);
``copes`` is its thin ctypes binding, and ``workloads`` describes the seeded synthetic
workloads.  Importing the package does not load the library; ``copes.load()`` (called by
every binding function) does, and raises if it is missing.
"""
__all__ = ["copes", "workloads"]
