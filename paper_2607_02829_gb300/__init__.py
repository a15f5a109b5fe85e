"""GB300-native Sparse-Reslim routed encoder forward (arxiv 2607.02829).

The computation lives in the CUDA library ``libsparse_reslim.so`` (sources in
``csrc/``, C ABI in ``include/sparse_reslim.h``); ``binding`` is its ctypes
binding and ``synth`` the seeded synthetic-input generator.  The library is
loaded on first use and its absence is an error.
"""
