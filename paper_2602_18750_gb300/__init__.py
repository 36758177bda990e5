"""GB300-native token-importance evaluation for KV eviction (HillInfer, arxiv 2602.18750).

Layout:
  csrc/      CUDA kernels for sm_103a and the C ABI (libhill.so)
  hill.py    thin ctypes binding over the C ABI (same names: hill_score, ...)
  build.py   nvcc build of libhill.so
  inputs.py  seeded synthetic workloads (no evaluation arithmetic)

Importing the package does not load the CUDA library; ``hill`` does, and it
raises if the library is missing.
"""
