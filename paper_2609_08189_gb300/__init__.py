"""GB300 (sm_103a) implementation of HeRo's history-aware routed FFN stack.

The compute path is libhero.so (hand-written CUDA kernels behind the C ABI of
include/hero.h); `paper_2609_08189_gb300.hero` is its ctypes binding.
"""
