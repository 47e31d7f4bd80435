"""GB300-native batched inference of the bidirectional minGRU track-fit encoder.

The compute path is the C-ABI library built from ``csrc/`` (see
``include/trackfit.h``); ``trackfit`` is its thin ctypes binding and
``workloads`` the seeded synthetic inputs.  Importing the package loads nothing:
``trackfit.load()`` opens the library and fails loudly if it is missing.
"""
__all__ = ["workloads", "trackfit"]
