"""GB300-native region-sparse DiT denoising step (RegionCache).

The compute path lives in the CUDA library built from ``csrc/`` and is reached
through the C ABI declared in ``include/regioncache.h``; ``regioncache`` is the
thin ctypes binding with the same entry-point names.  ``synth`` draws the
seeded synthetic workloads.
"""
__all__ = ["synth"]
