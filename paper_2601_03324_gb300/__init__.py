"""GB300-native batch-1 FP32 decode of a Llama-2-architecture decoder.

The compute path is hand-written CUDA for sm_103a behind the C ABI declared in
``include/tvl.h`` (library ``libtvl.so``); :mod:`.tvl` is a thin ctypes
binding over it and :mod:`.synth` makes seeded synthetic inputs.
"""
__all__ = ["tvl", "synth"]
