"""GB300 (sm_103a) packed LM-head forward of ARCHead.

The compute path lives in libarchead.so (CUDA kernels behind a C ABI,
include/archead.h); ``archead`` is its thin ctypes binding and ``build``
compiles it with nvcc.
"""

from . import archead  # noqa: F401
from . import build as _build_module  # noqa: F401
