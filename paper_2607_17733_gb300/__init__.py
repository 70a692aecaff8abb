"""MXINT mixed-precision linear layer (MXSens, arxiv 2607.17733) for GB300 / sm_103a.

The compute path is libmxs.so (hand-written CUDA behind a C ABI, declared in
include/mxs.h); `paper_2607_17733_gb300.mxs` is a thin ctypes binding over it.
Importing this package does not load the library; the first call does, and
it raises if the library is missing -- there is no CPU fallback.
"""
