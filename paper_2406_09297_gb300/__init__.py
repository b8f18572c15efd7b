"""GB300-native MLKV decode attention (arXiv 2406.09297).

The library is libmlkv.so (C ABI in include/mlkv.h, CUDA kernels for sm_103a); ``mlkv`` is its
Python binding.  Build with ``paper_2406_09297_gb300.build.build()``.
"""
from .mlkv import *  # noqa: F401,F403
from .mlkv import MLKVCache, MLKVError  # noqa: F401
