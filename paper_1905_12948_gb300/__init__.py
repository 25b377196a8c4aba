"""GB300 (sm_103a) implementation of one Global Momentum Compression step
(GMC / GMC+, arXiv 1905.12948) for K data-parallel workers simulated on one GPU.

The method runs in the CUDA kernels of ``libgmc.so`` behind the C ABI of
``include/gmc.h``; ``gmc`` is its Python binding.
"""
from .gmc import GMC, GMCError, load  # noqa: F401
