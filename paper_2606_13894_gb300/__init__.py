"""GB300-native (sm_103a) implementation of the Gefen optimizer's hot path.

Gefen (arXiv 2606.13894) shares one second moment per automatically inferred
parameter block (Algorithm 2) and stores the first moment as 8-bit codes of a
learned codebook (Algorithm 3) scaled by the block's absmax (Algorithm 1).

The compute path is the C-ABI library ``libgefen.so`` (hand-written CUDA for
sm_103a, declared in ``include/gefen.h``); :mod:`.gefen` is its thin ctypes
binding.  Importing this package loads nothing: the library is opened on the
first call, and every entry point raises if it is missing.
"""
__all__ = ["gefen", "synth"]
