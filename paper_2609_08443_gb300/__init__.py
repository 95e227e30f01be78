"""GB300-native Sketch Attention sketching step (SequenceO1, Sec. 3.1 and Sec. 4.4).

The compute lives in ``libsa_sketch.so`` (hand-written sm_103a CUDA behind a
C ABI declared in ``include/sa_sketch.h``); ``binding`` is a thin ctypes layer
that passes torch's device pointers and current stream to it.  The library is
loaded lazily on first use and its absence is an error, never a fallback.
"""
__all__ = ["binding", "workloads", "roofline"]
