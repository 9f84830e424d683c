"""K-interval attention (forward and backward) on NVIDIA GB300, sm_103a.

The operator lives in the C-ABI library libkint (include/kint_attn.h, sources
in csrc/); ``kint`` is its Python binding and ``inputs`` the seeded synthetic
input generator.
"""
