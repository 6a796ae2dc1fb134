"""GB300-native Shift Sparse Block Attention (SSBA) forward.

The compute path is the CUDA library ``libssba.so`` (hand-written sm_103a kernels
behind the C-ABI declared in ``include/ssba.h``); this package is a thin ctypes
binding over it. There is no CPU fallback: if the library is missing the calls
raise.
"""
from .api import (  # noqa: F401
    SsbaDesc, SsbaError, BoundLayer, BoundSelectLayer, backward, backward_workspace_bytes, build_mask,
    build_mask_noalloc, default_forward_workspace, forward, forward_dense, forward_fused, forward_joint,
    forward_select, forward_workspace_bytes, get_status, haar_dwt, haar_dwt_pyramid, haar_iwt, haar_iwt_pyramid,
    keep_count, library_path, load_library, mask_workspace_bytes, pool_blocks, qkv_rope_pool, realized_sparsity,
    select_mask,
)

__all__ = [
    "SsbaDesc", "SsbaError", "BoundLayer", "BoundSelectLayer", "backward", "backward_workspace_bytes",
    "build_mask", "build_mask_noalloc", "default_forward_workspace", "forward", "forward_dense", "forward_fused",
    "forward_joint", "forward_select", "forward_workspace_bytes", "get_status", "haar_dwt", "haar_dwt_pyramid",
    "haar_iwt", "haar_iwt_pyramid", "keep_count", "library_path", "load_library", "mask_workspace_bytes",
    "pool_blocks", "qkv_rope_pool", "realized_sparsity", "select_mask",
]
