"""GB300-native chunkwise gated-linear-attention forward (the GTR token mixer).

The compute path is a C-ABI shared library of hand-written sm_103a CUDA
kernels (``csrc/``, declared in ``include/gtr_gla.h``); :mod:`.gla` is the thin
ctypes binding over it and uses PyTorch only for device memory and streams.
:mod:`.workloads` draws the seeded synthetic inputs.
"""
__all__ = ["gla", "workloads"]
