"""GB300-native batched multi-draft speculative verification.

Hot path: hand-written sm_103a CUDA in ``csrc/`` behind the C ABI of
``include/mds.h``; ``mds`` is the ctypes binding (import it after building
the library with ``build.build()``).
"""
__all__ = ["build", "mds"]
