"""GB300-native LittleBit linear forward (arXiv 2506.13771).

The compute lives in the C-ABI library ``liblittlebit.so`` (hand-written
sm_103a CUDA under ``csrc/``, declared in ``include/littlebit.h``).
``littlebit`` is the thin ctypes binding over it; ``inputs`` draws the seeded
synthetic workloads.  Importing the package does not load the library: the
binding loads it on first use and raises if it is missing.
"""
__all__ = ["inputs", "littlebit"]
