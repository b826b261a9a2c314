"""GB300 (sm_103a) implementation of SPHQuant's fused spherical dequantize-GEMV.

The compute lives in libsphq.so (C ABI: include/sphq.h); ``sphq`` is its thin
Python binding.
"""
from .sphq import SphqError, SphqMatrix, header_functions, load  # noqa: F401
