"""GB300 (sm_103a) implementation of the inference hot path of Elastic
Significant Bit quantization (Gong et al., arXiv 2109.03513).

The compute path is the C-ABI library ``libesb.so`` (CUDA kernels in
``csrc/``, interface in ``include/esb.h``); ``esb`` is its ctypes binding.
"""
from . import esb  # noqa: F401  (the binding loads libesb.so lazily, on first call)

__all__ = ["esb"]
