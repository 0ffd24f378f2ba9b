"""GB300-native (sm_103a) Dynamic Linear Attention forward path.

The compute lives in the C-ABI library ``libdla.so`` built from ``csrc/``
(hand-written CUDA); :mod:`.dla` is the thin ctypes binding with the same
entry-point names as ``include/dla.h``; :mod:`.workloads` holds the seeded
synthetic inputs.
"""
