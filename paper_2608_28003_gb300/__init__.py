"""GB300 (sm_103a) implementation of the W8A8 SmoothQuant hot path of arXiv 2608.28003.

The compute lives in ``libw8a8.so`` (CUDA kernels behind the C ABI of ``include/w8a8.h``);
``binding`` is a ctypes layer that marshals torch tensors into that ABI.  Build the library
with ``paper_2608_28003_gb300.build.build()``.
"""
from . import binding  # noqa: F401
from .binding import W8A8_PREC_BF16, W8A8_PREC_W8A8, W8A8Error  # noqa: F401
