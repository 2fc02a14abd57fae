"""GB300-native (sm_103a) EAT MoE-layer hot path behind a C ABI (libeat.so).

The compute path lives in ``csrc/`` (CUDA kernels + the extern "C" boundary declared in
``include/eat.h``); ``eat`` is the thin ctypes binding with the same names.  The shared library is
loaded on first use and its absence is an error: there is no CPU fallback.
"""
