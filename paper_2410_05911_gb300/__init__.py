"""GB300 (sm_103a) implementation of the AECCT batched inference forward pass.

The decoder runs in libaecct.so (C ABI in include/aecct.h); `aecct` is its Python binding
and `inputs` builds seeded synthetic codes, channel outputs and model tensors.
"""
__all__ = ["aecct", "inputs", "build_lib"]
