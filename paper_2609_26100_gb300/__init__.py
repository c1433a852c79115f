"""GB300-native TSS target-side verification: a C-ABI CUDA library plus a thin ctypes binding.

The library (``libtss.so``, built from ``csrc/``) runs the verification forward pass of a LLaMA
decoder under a per-domain layer-skip mask, then greedy or speculative-sampling acceptance and KV
compaction, all in hand-written sm_103a kernels.  ``synth`` draws seeded synthetic inputs.
"""
__all__ = ["synth"]
