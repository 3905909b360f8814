"""GB300-native (sm_103a) ABCD active-block hot path.

The compute lives in ``libabcd.so`` (hand-written CUDA behind a C ABI, declared in
``include/abcd.h``); this package is a thin ctypes binding with the same names.
"""
