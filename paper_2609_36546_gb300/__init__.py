"""GB300-native (sm_103a) verify step of Interactive-Policy Distillation.

The compute runs in libipd.so (hand-written CUDA behind the C ABI of
include/ipd.h); this package is its Python binding (``ipd``) and the host
glue that assembles one step (``step``).  Importing it fails loudly when the
library has not been built.
"""
from . import ipd  # noqa: F401
from .ipd import IpdError  # noqa: F401
from .step import VerifyStep  # noqa: F401

__all__ = ["ipd", "IpdError", "VerifyStep"]
