"""GB300-native Deep Parity Bottleneck (DPB): encode, decode and backward.

The compute path is the C-ABI library ``libdpb.so`` (hand-written sm_103a
CUDA kernels behind ``include/dpb.h``); ``paper_2607_20652_gb300.dpb`` is a
thin ctypes binding with the same entry-point names. Importing this package
does not load the library; the first call through ``dpb`` does, and fails
loudly if it is missing.
"""
