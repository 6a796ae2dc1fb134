"""GB300-native Shift Sparse Block Attention (SSBA) forward.

The compute path is the CUDA library ``libssba.so`` (hand-written sm_103a kernels
behind the C-ABI declared in ``include/ssba.h``); this package is a thin ctypes
binding over it. There is no CPU fallback: if the library is missing the calls
raise.
"""
from .api import (  # noqa: F401
    SsbaDesc, SsbaError, build_mask, forward, forward_dense, keep_count, mask_workspace_bytes,
    get_status, library_path, load_library,
)

__all__ = [
    "SsbaDesc", "SsbaError", "build_mask", "forward", "forward_dense", "keep_count",
    "mask_workspace_bytes", "get_status", "library_path", "load_library",
]
