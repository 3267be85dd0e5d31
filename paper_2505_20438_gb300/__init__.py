"""GB300-native smashed-KV decode attention (HAMburger, arXiv 2505.20438).

The compute path is libham.so (C ABI in include/ham.h, CUDA kernels for sm_103a under
csrc/); `ham` is its Python binding and `workload` draws seeded synthetic inputs.
"""
