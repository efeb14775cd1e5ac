"""libkvrepair: budgeted in-place repair of stale KV caches on GB300 (sm_103a).

The compute path is the C-ABI shared library ``libkvrepair.so`` (CUDA kernels
in ``csrc/``), reached from Python through ``kvrepair`` (ctypes marshalling
only).  ``synth`` generates seeded synthetic inputs.  Importing this package
loads nothing; importing ``kvrepair`` loads the library and fails loudly if it
has not been built.
"""
__all__ = ["kvrepair", "synth"]
