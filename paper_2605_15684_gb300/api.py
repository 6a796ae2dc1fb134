"""ctypes binding of libssba.so (include/ssba.h), same names as the C entry points.

Argument marshalling only: tensors are checked for device, dtype, shape and
contiguity, their ``data_ptr()`` and the current CUDA stream are handed to the C
call, and a non-zero status is raised as ``SsbaError``. Every step of the path
runs in the library's kernels; there is no Python or CPU fallback, and the
library must exist (``paper_2605_15684_gb300.build.build()`` makes it).
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libssba.so")
_lock = threading.Lock()
_lib = None

(SSBA_OK, SSBA_ERR_INVALID, SSBA_ERR_UNSUPPORTED, SSBA_ERR_CUDA, SSBA_ERR_TIMEOUT, SSBA_ERR_WORKSPACE,
 SSBA_ERR_CHECK) = range(7)
SSBA_BF16, SSBA_FP32 = 0, 1
_STATUS_NAMES = {0: "SSBA_OK", 1: "SSBA_ERR_INVALID", 2: "SSBA_ERR_UNSUPPORTED", 3: "SSBA_ERR_CUDA",
                 4: "SSBA_ERR_TIMEOUT", 5: "SSBA_ERR_WORKSPACE", 6: "SSBA_ERR_CHECK"}

EXPORTED = ("ssba_keep_count", "ssba_mask_workspace_bytes", "ssba_build_mask", "ssba_build_mask_noalloc",
            "ssba_forward", "ssba_forward_joint", "ssba_forward_workspace_bytes", "ssba_forward_dense",
            "ssba_test_forward_timeout", "ssba_test_fused_timeout", "ssba_test_backward_timeout", "ssba_backward", "ssba_backward_workspace_bytes", "ssba_haar_dwt",
            "ssba_haar_iwt", "ssba_haar_dwt_pyramid", "ssba_haar_iwt_pyramid", "ssba_qkv_rope_pool",
            "ssba_select_mask", "ssba_pool_blocks", "ssba_forward_select", "ssba_forward_fused",
            "ssba_get_status", "ssba_last_error", "ssba_timeline_read")


class SsbaError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{_STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


class _Desc(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("heads", ctypes.c_int32), ("H_tok", ctypes.c_int32),
                ("W_tok", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("block", ctypes.c_int32),
                ("shift_r", ctypes.c_int32), ("shift_c", ctypes.c_int32), ("rho", ctypes.c_double),
                ("dtype", ctypes.c_int32), ("softmax_scale", ctypes.c_float)]


@dataclass
class SsbaDesc:
    """Python mirror of ``ssba_desc``."""
    B: int
    heads: int
    H_tok: int
    W_tok: int
    head_dim: int = 64
    block: int = 8
    shift_r: int = 0
    shift_c: int = 0
    rho: float = 0.0
    dtype: torch.dtype = torch.bfloat16
    softmax_scale: float = 0.0

    @property
    def N(self) -> int:
        return self.H_tok * self.W_tok

    @property
    def Tb(self) -> int:
        return self.N // (self.block * self.block)

    def c(self) -> _Desc:
        if self.dtype == torch.bfloat16:
            dt = SSBA_BF16
        elif self.dtype == torch.float32:
            dt = SSBA_FP32
        else:
            raise SsbaError(SSBA_ERR_INVALID, f"unsupported dtype {self.dtype}")
        return _Desc(self.B, self.heads, self.H_tok, self.W_tok, self.head_dim, self.block,
                     self.shift_r, self.shift_c, float(self.rho), dt, float(self.softmax_scale))


def library_path() -> str:
    return _LIB_PATH


def load_library(path: str | None = None):
    """Load libssba.so (raises if it has not been built). ``path`` selects another build of
    the same library (the timeline or checked variant of build.py) on the first call; every
    later call returns the library loaded first."""
    global _lib, _LIB_PATH
    with _lock:
        if _lib is not None:
            if path is not None and os.path.abspath(path) != _LIB_PATH:
                raise SsbaError(SSBA_ERR_INVALID, f"{_LIB_PATH} is already loaded in this process")
            return _lib
        if path is not None:
            _LIB_PATH = os.path.abspath(path)
        if not os.path.exists(_LIB_PATH):
            raise SsbaError(SSBA_ERR_CUDA, f"{_LIB_PATH} is missing: run paper_2605_15684_gb300.build.build()")
        lib = ctypes.CDLL(_LIB_PATH)
        P = ctypes.c_void_p
        DP = ctypes.POINTER(_Desc)
        lib.ssba_keep_count.argtypes = [DP]
        lib.ssba_keep_count.restype = ctypes.c_int
        lib.ssba_mask_workspace_bytes.argtypes = [DP]
        lib.ssba_mask_workspace_bytes.restype = ctypes.c_size_t
        lib.ssba_build_mask.argtypes = [DP, P, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_build_mask.restype = ctypes.c_int
        lib.ssba_build_mask_noalloc.argtypes = [DP, P, P, P, P, P, P]
        lib.ssba_build_mask_noalloc.restype = ctypes.c_int
        lib.ssba_qkv_rope_pool.argtypes = [DP, P, P, P, P, P, P, P, P, P]
        lib.ssba_qkv_rope_pool.restype = ctypes.c_int
        lib.ssba_select_mask.argtypes = [DP, P, P, P, P, P, P]
        lib.ssba_select_mask.restype = ctypes.c_int
        lib.ssba_pool_blocks.argtypes = [DP, P, P, P, P, P]
        lib.ssba_pool_blocks.restype = ctypes.c_int
        lib.ssba_forward_select.argtypes = [DP, P, P, P, P, P, P, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_forward_select.restype = ctypes.c_int
        lib.ssba_forward_fused.argtypes = [DP, P, P, P, P, P, P, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_forward_fused.restype = ctypes.c_int
        lib.ssba_forward.argtypes = [DP, P, P, P, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_forward.restype = ctypes.c_int
        lib.ssba_forward_joint.argtypes = [DP, P, P, P, P, P, ctypes.c_int32, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_forward_joint.restype = ctypes.c_int
        lib.ssba_forward_workspace_bytes.argtypes = [DP]
        lib.ssba_forward_workspace_bytes.restype = ctypes.c_size_t
        lib.ssba_forward_dense.argtypes = [DP, P, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_forward_dense.restype = ctypes.c_int
        lib.ssba_test_forward_timeout.argtypes = [DP, P, P, P, P, P, P, P, ctypes.c_uint64, P]
        lib.ssba_test_forward_timeout.restype = ctypes.c_int
        lib.ssba_test_fused_timeout.argtypes = [DP, P, P, P, P, P, P, P, P, P, P, ctypes.c_size_t, ctypes.c_uint64, P]
        lib.ssba_test_fused_timeout.restype = ctypes.c_int
        lib.ssba_backward.argtypes = [DP, P, P, P, P, P, P, P, P, P, P, P, P, ctypes.c_size_t, P]
        lib.ssba_backward.restype = ctypes.c_int
        lib.ssba_test_backward_timeout.argtypes = [DP, P, P, P, P, P, P, P, P, P, P, P, P, ctypes.c_size_t,
                                                   ctypes.c_uint64, P]
        lib.ssba_test_backward_timeout.restype = ctypes.c_int
        lib.ssba_backward_workspace_bytes.argtypes = [DP]
        lib.ssba_backward_workspace_bytes.restype = ctypes.c_size_t
        I = ctypes.c_int32
        for fn in ("ssba_haar_dwt", "ssba_haar_iwt"):
            getattr(lib, fn).argtypes = [P, P, I, I, I, I, I, I, P]
            getattr(lib, fn).restype = ctypes.c_int
        PP = ctypes.POINTER(ctypes.c_void_p)
        lib.ssba_haar_dwt_pyramid.argtypes = [P, PP, I, I, I, I, I, I, I, P]
        lib.ssba_haar_dwt_pyramid.restype = ctypes.c_int
        lib.ssba_haar_iwt_pyramid.argtypes = [PP, P, I, I, I, I, I, I, I, P]
        lib.ssba_haar_iwt_pyramid.restype = ctypes.c_int
        lib.ssba_get_status.argtypes = [ctypes.POINTER(ctypes.c_int32)]
        lib.ssba_get_status.restype = ctypes.c_int
        lib.ssba_last_error.argtypes = []
        lib.ssba_last_error.restype = ctypes.c_char_p
        lib.ssba_timeline_read.argtypes = [P, P, P]
        lib.ssba_timeline_read.restype = ctypes.c_int
        _lib = lib
        return lib


def _raise_on(rc: int) -> None:
    if rc != SSBA_OK:
        raise SsbaError(rc, _lib.ssba_last_error().decode(errors="replace"))


def _stream_ptr(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _check(t: torch.Tensor, name: str, shape, dtype) -> None:
    if not isinstance(t, torch.Tensor):
        raise SsbaError(SSBA_ERR_INVALID, f"{name} must be a torch.Tensor")
    if t.device.type != "cuda":
        raise SsbaError(SSBA_ERR_INVALID, f"{name} must be a CUDA tensor (got {t.device})")
    if tuple(t.shape) != tuple(shape):
        raise SsbaError(SSBA_ERR_INVALID, f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    if t.dtype != dtype:
        raise SsbaError(SSBA_ERR_INVALID, f"{name} has dtype {t.dtype}, expected {dtype}")
    if not t.is_contiguous():
        raise SsbaError(SSBA_ERR_INVALID, f"{name} must be contiguous")


def keep_count(desc: SsbaDesc) -> int:
    lib = load_library()
    d = desc.c()
    k = lib.ssba_keep_count(ctypes.byref(d))
    if k < 0:
        _raise_on(SSBA_ERR_INVALID)
    return k


def mask_workspace_bytes(desc: SsbaDesc) -> int:
    lib = load_library()
    d = desc.c()
    return int(lib.ssba_mask_workspace_bytes(ctypes.byref(d)))


def forward_workspace_bytes(desc: SsbaDesc) -> int:
    lib = load_library()
    d = desc.c()
    return int(lib.ssba_forward_workspace_bytes(ctypes.byref(d)))


_fwd_ws: dict = {}


def default_forward_workspace(desc: SsbaDesc, device, stream=None) -> torch.Tensor:
    """A zero-filled forward workspace kept per (device, stream) and reused by every call on
    that stream that passes none (``stream`` None: the current stream). The kernels leave it
    zero-filled, so the calls of one stream, which run in order, can share it; calls on two
    streams get two workspaces, so they never share its counters or barrier words."""
    need = forward_workspace_bytes(desc)
    dev = torch.device(device)
    idx = dev.index if dev.index is not None else torch.cuda.current_device()
    with torch.cuda.device(idx):
        key = (idx, _stream_ptr(stream))
    with _lock:
        ws = _fwd_ws.get(key)
        if ws is None or ws.numel() < need:
            ws = torch.zeros(max(need, 1), dtype=torch.uint8, device=dev)
            _fwd_ws[key] = ws
    return ws


def _ws_args(ws):
    if ws is None:
        return None, 0
    if not isinstance(ws, torch.Tensor) or ws.device.type != "cuda" or not ws.is_contiguous():
        raise SsbaError(SSBA_ERR_INVALID, "workspace must be a contiguous CUDA tensor")
    return ws.data_ptr(), ws.numel() * ws.element_size()


def build_mask(desc: SsbaDesc, Q: torch.Tensor, K: torch.Tensor, kv_idx=None, kv_cnt=None,
               scores: bool | torch.Tensor = False, workspace=None, stream=None):
    """ssba_build_mask: returns (kv_idx [B,h,Tb,keep] int32, kv_cnt [B,h,Tb] int32[, S])."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    _check(Q, "Q", shp, desc.dtype)
    _check(K, "K", shp, desc.dtype)
    dev = Q.device
    if kv_idx is None:
        kv_idx = torch.empty((desc.B, desc.heads, desc.Tb, keep), dtype=torch.int32, device=dev)
    if kv_cnt is None:
        kv_cnt = torch.empty((desc.B, desc.heads, desc.Tb), dtype=torch.int32, device=dev)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    S = None
    if isinstance(scores, torch.Tensor):
        S = scores
        _check(S, "scores", (desc.B, desc.heads, desc.Tb, desc.Tb), torch.float32)
    elif scores:
        S = torch.empty((desc.B, desc.heads, desc.Tb, desc.Tb), dtype=torch.float32, device=dev)
    ws_need = int(lib.ssba_mask_workspace_bytes(ctypes.byref(d)))
    if workspace is None:
        workspace = torch.empty(ws_need, dtype=torch.uint8, device=dev)
    rc = lib.ssba_build_mask(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), kv_idx.data_ptr(),
                             kv_cnt.data_ptr(), S.data_ptr() if S is not None else None,
                             workspace.data_ptr(), workspace.numel() * workspace.element_size(),
                             _stream_ptr(stream))
    _raise_on(rc)
    return (kv_idx, kv_cnt, S) if S is not None else (kv_idx, kv_cnt)


def qkv_rope_pool(desc: SsbaDesc, X: torch.Tensor, Wqkv: torch.Tensor, bias=None, pooled: bool = True,
                  out=None, stream=None):
    """ssba_qkv_rope_pool: X [B, N, heads*64] -> (Q, K, V [B, heads, N, 64] bf16 with RoPE on Q
    and K, qb, kb [B, heads, Tb, 64] fp32 block means, or None when pooled is False)."""
    lib = load_library()
    d = desc.c()
    Dm = desc.heads * desc.head_dim
    _check(X, "X", (desc.B, desc.N, Dm), torch.bfloat16)
    _check(Wqkv, "Wqkv", (3 * Dm, Dm), torch.bfloat16)
    if bias is not None:
        _check(bias, "bias", (3 * Dm,), torch.float32)
    dev = X.device
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    pshp = (desc.B, desc.heads, desc.Tb, desc.head_dim)
    if out is None:
        out = [torch.empty(shp, dtype=torch.bfloat16, device=dev) for _ in range(3)]
        out += [torch.empty(pshp, dtype=torch.float32, device=dev) for _ in range(2)] if pooled else [None, None]
    Q, K, V, qb, kb = out
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _check(t, n, shp, torch.bfloat16)
    for t, n in ((qb, "qb"), (kb, "kb")):
        if t is not None:
            _check(t, n, pshp, torch.float32)
    _raise_on(lib.ssba_qkv_rope_pool(ctypes.byref(d), X.data_ptr(), Wqkv.data_ptr(),
                                     bias.data_ptr() if bias is not None else None, Q.data_ptr(), K.data_ptr(),
                                     V.data_ptr(), qb.data_ptr() if qb is not None else None,
                                     kb.data_ptr() if kb is not None else None, _stream_ptr(stream)))
    return Q, K, V, qb, kb


def select_mask(desc: SsbaDesc, qb: torch.Tensor, kb: torch.Tensor, kv_idx=None, kv_cnt=None,
                scores: bool | torch.Tensor = False, stream=None):
    """ssba_select_mask: block means -> (kv_idx, kv_cnt[, S]) as build_mask returns them."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    pshp = (desc.B, desc.heads, desc.Tb, desc.head_dim)
    _check(qb, "qb", pshp, torch.float32)
    _check(kb, "kb", pshp, torch.float32)
    dev = qb.device
    if kv_idx is None:
        kv_idx = torch.empty((desc.B, desc.heads, desc.Tb, keep), dtype=torch.int32, device=dev)
    if kv_cnt is None:
        kv_cnt = torch.empty((desc.B, desc.heads, desc.Tb), dtype=torch.int32, device=dev)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    S = None
    if isinstance(scores, torch.Tensor):
        S = scores
        _check(S, "scores", (desc.B, desc.heads, desc.Tb, desc.Tb), torch.float32)
    elif scores:
        S = torch.empty((desc.B, desc.heads, desc.Tb, desc.Tb), dtype=torch.float32, device=dev)
    _raise_on(lib.ssba_select_mask(ctypes.byref(d), qb.data_ptr(), kb.data_ptr(), kv_idx.data_ptr(),
                                   kv_cnt.data_ptr(), S.data_ptr() if S is not None else None, _stream_ptr(stream)))
    return (kv_idx, kv_cnt, S) if S is not None else (kv_idx, kv_cnt)


def pool_blocks(desc: SsbaDesc, Q: torch.Tensor, K: torch.Tensor, qb=None, kb=None, stream=None):
    """ssba_pool_blocks: (qb, kb) fp32 [B, heads, Tb, head_dim] block means of Q and K."""
    lib = load_library()
    d = desc.c()
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    _check(Q, "Q", shp, desc.dtype)
    _check(K, "K", shp, desc.dtype)
    pshp = (desc.B, desc.heads, desc.Tb, desc.head_dim)
    qb = torch.empty(pshp, dtype=torch.float32, device=Q.device) if qb is None else qb
    kb = torch.empty(pshp, dtype=torch.float32, device=Q.device) if kb is None else kb
    _check(qb, "qb", pshp, torch.float32)
    _check(kb, "kb", pshp, torch.float32)
    _raise_on(lib.ssba_pool_blocks(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), qb.data_ptr(), kb.data_ptr(),
                                   _stream_ptr(stream)))
    return qb, kb


def _forward_select_call(fn_name, desc, Q, K, V, qb, kb, kv_idx, kv_cnt, scores, O, lse, workspace, stream):
    lib = load_library()
    d = desc.c()
    keep = keep_count(desc)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _check(t, n, shp, desc.dtype)
    dev = Q.device
    pshp = (desc.B, desc.heads, desc.Tb, desc.head_dim)
    qb = torch.empty(pshp, dtype=torch.float32, device=dev) if qb is None else qb
    kb = torch.empty(pshp, dtype=torch.float32, device=dev) if kb is None else kb
    _check(qb, "qb", pshp, torch.float32)
    _check(kb, "kb", pshp, torch.float32)
    kv_idx = torch.empty((desc.B, desc.heads, desc.Tb, keep), dtype=torch.int32, device=dev) if kv_idx is None \
        else kv_idx
    kv_cnt = torch.empty((desc.B, desc.heads, desc.Tb), dtype=torch.int32, device=dev) if kv_cnt is None else kv_cnt
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    S = None
    if isinstance(scores, torch.Tensor):
        S = scores
        _check(S, "scores", (desc.B, desc.heads, desc.Tb, desc.Tb), torch.float32)
    elif scores:
        S = torch.empty((desc.B, desc.heads, desc.Tb, desc.Tb), dtype=torch.float32, device=dev)
    O = torch.empty(shp, dtype=desc.dtype, device=dev) if O is None else O
    lse = torch.empty(shp[:3], dtype=torch.float32, device=dev) if lse is None else lse
    _check(O, "O", shp, desc.dtype)
    _check(lse, "lse", shp[:3], torch.float32)
    if isinstance(workspace, str):
        workspace = default_forward_workspace(desc, dev, stream)
    wp, wn = _ws_args(workspace)
    _raise_on(getattr(lib, fn_name)(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), qb.data_ptr(),
                                    kb.data_ptr(), kv_idx.data_ptr(), kv_cnt.data_ptr(),
                                    S.data_ptr() if S is not None else None, O.data_ptr(), lse.data_ptr(), wp, wn,
                                    _stream_ptr(stream)))
    return qb, kb, kv_idx, kv_cnt, S, O, lse


def forward_select(desc: SsbaDesc, Q, K, V, qb, kb, kv_idx=None, kv_cnt=None, scores: bool | torch.Tensor = False,
                   O=None, lse=None, workspace="default", stream=None):
    """ssba_forward_select: selection inside the attention launch. Returns (O, lse, kv_idx, kv_cnt[, S])."""
    if qb is None or kb is None:
        raise SsbaError(SSBA_ERR_INVALID, "forward_select needs the block means qb, kb")
    _, _, kv_idx, kv_cnt, S, O, lse = _forward_select_call("ssba_forward_select", desc, Q, K, V, qb, kb, kv_idx,
                                                           kv_cnt, scores, O, lse, workspace, stream)
    return (O, lse, kv_idx, kv_cnt, S) if S is not None else (O, lse, kv_idx, kv_cnt)


def forward_fused(desc: SsbaDesc, Q, K, V, qb=None, kb=None, kv_idx=None, kv_cnt=None,
                  scores: bool | torch.Tensor = False, O=None, lse=None, workspace="default", stream=None):
    """ssba_forward_fused: pooling, selection and attention in one launch.
    Returns (O, lse, kv_idx, kv_cnt, qb, kb[, S])."""
    if workspace is None:
        raise SsbaError(SSBA_ERR_WORKSPACE, "forward_fused needs a forward workspace")
    qb, kb, kv_idx, kv_cnt, S, O, lse = _forward_select_call("ssba_forward_fused", desc, Q, K, V, qb, kb, kv_idx,
                                                             kv_cnt, scores, O, lse, workspace, stream)
    return (O, lse, kv_idx, kv_cnt, qb, kb, S) if S is not None else (O, lse, kv_idx, kv_cnt, qb, kb)


def build_mask_noalloc(desc: SsbaDesc, Q: torch.Tensor, K: torch.Tensor, kv_idx=None, kv_cnt=None,
                       scores: bool | torch.Tensor = False, stream=None):
    """ssba_build_mask_noalloc: build_mask with the library's built-in scratch area (no
    workspace argument; see include/ssba.h for the size limit and the sharing rule)."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    _check(Q, "Q", shp, desc.dtype)
    _check(K, "K", shp, desc.dtype)
    dev = Q.device
    if kv_idx is None:
        kv_idx = torch.empty((desc.B, desc.heads, desc.Tb, keep), dtype=torch.int32, device=dev)
    if kv_cnt is None:
        kv_cnt = torch.empty((desc.B, desc.heads, desc.Tb), dtype=torch.int32, device=dev)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    S = None
    if isinstance(scores, torch.Tensor):
        S = scores
        _check(S, "scores", (desc.B, desc.heads, desc.Tb, desc.Tb), torch.float32)
    elif scores:
        S = torch.empty((desc.B, desc.heads, desc.Tb, desc.Tb), dtype=torch.float32, device=dev)
    rc = lib.ssba_build_mask_noalloc(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), kv_idx.data_ptr(),
                                     kv_cnt.data_ptr(), S.data_ptr() if S is not None else None,
                                     _stream_ptr(stream))
    _raise_on(rc)
    return (kv_idx, kv_cnt, S) if S is not None else (kv_idx, kv_cnt)


def forward(desc: SsbaDesc, Q, K, V, kv_idx, kv_cnt, O=None, lse=None, workspace="default", stream=None):
    """ssba_forward: returns (O [B,h,N,d] in desc.dtype, lse [B,h,N] fp32).
    ``workspace``: "default" (the per-stream one of default_forward_workspace), None (no
    workspace: whole-query-block shares) or a zero-filled uint8 CUDA tensor."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _check(t, n, shp, desc.dtype)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    if O is None:
        O = torch.empty(shp, dtype=desc.dtype, device=Q.device)
    if lse is None:
        lse = torch.empty(shp[:3], dtype=torch.float32, device=Q.device)
    _check(O, "O", shp, desc.dtype)
    _check(lse, "lse", shp[:3], torch.float32)
    if isinstance(workspace, str):
        workspace = default_forward_workspace(desc, Q.device, stream) if desc.dtype == torch.bfloat16 else None
    wp, wn = _ws_args(workspace)
    rc = lib.ssba_forward(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), kv_idx.data_ptr(),
                          kv_cnt.data_ptr(), O.data_ptr(), lse.data_ptr(), wp, wn, _stream_ptr(stream))
    _raise_on(rc)
    return O, lse


def forward_joint(desc: SsbaDesc, Q, K, V, K_txt, V_txt, kv_idx, kv_cnt, O=None, lse=None, workspace="default",
                  stream=None):
    """ssba_forward_joint: image rows of the joint [text; image] attention (Algorithm 1 with
    its text segment). K_txt, V_txt: [B, heads, T_txt, d] bf16. Returns (O, lse) of the
    image tokens."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _check(t, n, shp, desc.dtype)
    T_txt = int(K_txt.shape[2]) if isinstance(K_txt, torch.Tensor) and K_txt.dim() == 4 else -1
    tshp = (desc.B, desc.heads, max(T_txt, 0), desc.head_dim)
    _check(K_txt, "K_txt", tshp, desc.dtype)
    _check(V_txt, "V_txt", tshp, desc.dtype)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    if O is None:
        O = torch.empty(shp, dtype=desc.dtype, device=Q.device)
    if lse is None:
        lse = torch.empty(shp[:3], dtype=torch.float32, device=Q.device)
    _check(O, "O", shp, desc.dtype)
    _check(lse, "lse", shp[:3], torch.float32)
    if isinstance(workspace, str):
        workspace = default_forward_workspace(desc, Q.device, stream) if desc.dtype == torch.bfloat16 else None
    wp, wn = _ws_args(workspace)
    rc = lib.ssba_forward_joint(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(),
                                K_txt.data_ptr() if T_txt > 0 else None, V_txt.data_ptr() if T_txt > 0 else None,
                                T_txt, kv_idx.data_ptr(), kv_cnt.data_ptr(), O.data_ptr(), lse.data_ptr(), wp, wn,
                                _stream_ptr(stream))
    _raise_on(rc)
    return O, lse


def forward_dense(desc: SsbaDesc, Q, K, V, O=None, lse=None, workspace="default", stream=None):
    """ssba_forward_dense: dense softmax attention from the same build (workspace as in forward)."""
    lib = load_library()
    d = desc.c()
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _check(t, n, shp, desc.dtype)
    if O is None:
        O = torch.empty(shp, dtype=desc.dtype, device=Q.device)
    if lse is None:
        lse = torch.empty(shp[:3], dtype=torch.float32, device=Q.device)
    _check(O, "O", shp, desc.dtype)
    _check(lse, "lse", shp[:3], torch.float32)
    if isinstance(workspace, str):
        workspace = default_forward_workspace(desc, Q.device, stream) if desc.dtype == torch.bfloat16 else None
    wp, wn = _ws_args(workspace)
    rc = lib.ssba_forward_dense(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), O.data_ptr(),
                                lse.data_ptr(), wp, wn, _stream_ptr(stream))
    _raise_on(rc)
    return O, lse


def test_forward_timeout(desc: SsbaDesc, Q, K, V, kv_idx, kv_cnt, O, lse, budget_ns: int = 2_000_000,
                         stream=None) -> None:
    """ssba_test_forward_timeout: the failure-detection test hook (see include/ssba.h)."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O")):
        _check(t, n, shp, desc.dtype)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    _check(lse, "lse", shp[:3], torch.float32)
    _raise_on(lib.ssba_test_forward_timeout(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(),
                                            kv_idx.data_ptr(), kv_cnt.data_ptr(), O.data_ptr(), lse.data_ptr(),
                                            int(budget_ns), _stream_ptr(stream)))


def test_fused_timeout(desc: SsbaDesc, Q, K, V, qb, kb, kv_idx, kv_cnt, O, lse, workspace,
                       budget_ns: int = 2_000_000, stream=None) -> None:
    """ssba_test_fused_timeout: the fused launch's failure-detection test hook (include/ssba.h)."""
    lib = load_library()
    d = desc.c()
    keep = keep_count(desc)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O")):
        _check(t, n, shp, desc.dtype)
    pshp = (desc.B, desc.heads, desc.Tb, desc.head_dim)
    _check(qb, "qb", pshp, torch.float32)
    _check(kb, "kb", pshp, torch.float32)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    _check(lse, "lse", shp[:3], torch.float32)
    wp, wn = _ws_args(workspace)
    if wp is None:
        raise SsbaError(SSBA_ERR_WORKSPACE, "test_fused_timeout needs a forward workspace")
    _raise_on(lib.ssba_test_fused_timeout(ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), qb.data_ptr(),
                                          kb.data_ptr(), kv_idx.data_ptr(), kv_cnt.data_ptr(), O.data_ptr(),
                                          lse.data_ptr(), wp, wn, int(budget_ns), _stream_ptr(stream)))


def backward_workspace_bytes(desc: SsbaDesc) -> int:
    lib = load_library()
    d = desc.c()
    return int(lib.ssba_backward_workspace_bytes(ctypes.byref(d)))


def backward(desc: SsbaDesc, Q, K, V, O, lse, dO, kv_idx, kv_cnt, dQ=None, dK=None, dV=None, workspace=None,
             stream=None, _timeout_budget_ns=None):
    """ssba_backward: gradients (dQ, dK, dV) in fp32 of the sparse forward for output gradient dO.
    With _timeout_budget_ns set it calls the failure-detection test hook ssba_test_backward_timeout
    instead (see include/ssba.h): the gradients are then undefined."""
    lib = load_library()
    d = desc.c()
    keep = lib.ssba_keep_count(ctypes.byref(d))
    if keep < 0:
        _raise_on(SSBA_ERR_INVALID)
    shp = (desc.B, desc.heads, desc.N, desc.head_dim)
    for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O"), (dO, "dO")):
        _check(t, n, shp, desc.dtype)
    _check(lse, "lse", shp[:3], torch.float32)
    _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
    _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
    outs = []
    for t, n in ((dQ, "dQ"), (dK, "dK"), (dV, "dV")):
        if t is None:
            t = torch.empty(shp, dtype=torch.float32, device=Q.device)
        _check(t, n, shp, torch.float32)
        outs.append(t)
    need = int(lib.ssba_backward_workspace_bytes(ctypes.byref(d)))
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=Q.device)
    wp, wn = _ws_args(workspace)
    args = (ctypes.byref(d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), O.data_ptr(), lse.data_ptr(), dO.data_ptr(),
            kv_idx.data_ptr(), kv_cnt.data_ptr(), outs[0].data_ptr(), outs[1].data_ptr(), outs[2].data_ptr(), wp, wn)
    if _timeout_budget_ns is None:
        rc = lib.ssba_backward(*args, _stream_ptr(stream))
    else:
        rc = lib.ssba_test_backward_timeout(*args, int(_timeout_budget_ns), _stream_ptr(stream))
    _raise_on(rc)
    return tuple(outs)


def test_backward_timeout(desc: SsbaDesc, Q, K, V, O, lse, dO, kv_idx, kv_cnt, budget_ns: int = 2_000_000,
                          stream=None) -> None:
    """ssba_test_backward_timeout: the backward's failure-detection test hook (include/ssba.h)."""
    backward(desc, Q, K, V, O, lse, dO, kv_idx, kv_cnt, stream=stream, _timeout_budget_ns=budget_ns)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return SSBA_BF16
    if t.dtype == torch.float32:
        return SSBA_FP32
    raise SsbaError(SSBA_ERR_INVALID, f"unsupported dtype {t.dtype}")


def haar_dwt(x: torch.Tensor, nb: int = 4, y=None, stream=None) -> torch.Tensor:
    """ssba_haar_dwt: x [N, C, H, W] -> [N, nb*C, H/2, W/2] (LL, HL, LH[, HH] bands)."""
    lib = load_library()
    if not isinstance(x, torch.Tensor) or x.dim() != 4:
        raise SsbaError(SSBA_ERR_INVALID, "x must be a 4-D tensor [N, C, H, W]")
    N, C, H, W = x.shape
    _check(x, "x", (N, C, H, W), x.dtype)
    if y is None:
        y = torch.empty((N, nb * C, H // 2, W // 2), dtype=x.dtype, device=x.device)
    _check(y, "y", (N, nb * C, H // 2, W // 2), x.dtype)
    _raise_on(lib.ssba_haar_dwt(x.data_ptr(), y.data_ptr(), N, C, H, W, nb, _dtype_code(x), _stream_ptr(stream)))
    return y


def haar_iwt(y: torch.Tensor, C: int, nb: int = 4, x=None, stream=None) -> torch.Tensor:
    """ssba_haar_iwt: y [N, nb*C, h, w] -> [N, C, 2h, 2w]."""
    lib = load_library()
    if not isinstance(y, torch.Tensor) or y.dim() != 4:
        raise SsbaError(SSBA_ERR_INVALID, "y must be a 4-D tensor [N, nb*C, h, w]")
    N, nbC, h, w = y.shape
    _check(y, "y", (N, nb * C, h, w), y.dtype)
    if x is None:
        x = torch.empty((N, C, 2 * h, 2 * w), dtype=y.dtype, device=y.device)
    _check(x, "x", (N, C, 2 * h, 2 * w), y.dtype)
    _raise_on(lib.ssba_haar_iwt(y.data_ptr(), x.data_ptr(), N, C, 2 * h, 2 * w, nb, _dtype_code(y), _stream_ptr(stream)))
    return x


HAAR_MAX_LEVELS = 3


def _ptr_array(ts):
    return (ctypes.c_void_p * len(ts))(*[t.data_ptr() for t in ts])


def haar_dwt_pyramid(x: torch.Tensor, levels: int, nb: int = 4, ys=None, stream=None):
    """ssba_haar_dwt_pyramid: x [N, C, H, W] -> [W1, ..., W_levels], W_l [N, nb*C, H/2^l, W/2^l]."""
    lib = load_library()
    if not isinstance(x, torch.Tensor) or x.dim() != 4:
        raise SsbaError(SSBA_ERR_INVALID, "x must be a 4-D tensor [N, C, H, W]")
    N, C, H, W = x.shape
    _check(x, "x", (N, C, H, W), x.dtype)
    if not 1 <= levels <= HAAR_MAX_LEVELS:
        raise SsbaError(SSBA_ERR_INVALID, f"levels must be 1..{HAAR_MAX_LEVELS}")
    shapes = [(N, nb * C, H >> l, W >> l) for l in range(1, levels + 1)]
    if ys is None:
        ys = [torch.empty(shp, dtype=x.dtype, device=x.device) for shp in shapes]
    if len(ys) != levels:
        raise SsbaError(SSBA_ERR_INVALID, f"ys must hold {levels} tensors")
    for l, (t, shp) in enumerate(zip(ys, shapes)):
        _check(t, f"ys[{l}]", shp, x.dtype)
    _raise_on(lib.ssba_haar_dwt_pyramid(x.data_ptr(), _ptr_array(ys), N, C, H, W, levels, nb, _dtype_code(x),
                                        _stream_ptr(stream)))
    return ys


def haar_iwt_pyramid(ys, C: int, nb: int = 4, x=None, stream=None) -> torch.Tensor:
    """ssba_haar_iwt_pyramid: [W1, ..., W_levels] -> x [N, C, H, W] (W1 is [N, nb*C, H/2, W/2])."""
    lib = load_library()
    levels = len(ys)
    if not 1 <= levels <= HAAR_MAX_LEVELS or not all(isinstance(t, torch.Tensor) and t.dim() == 4 for t in ys):
        raise SsbaError(SSBA_ERR_INVALID, f"ys must be 1..{HAAR_MAX_LEVELS} 4-D tensors")
    N, _, h, w = ys[0].shape
    H, W = 2 * h, 2 * w
    for l, t in enumerate(ys):
        _check(t, f"ys[{l}]", (N, nb * C, H >> (l + 1), W >> (l + 1)), ys[0].dtype)
    if x is None:
        x = torch.empty((N, C, H, W), dtype=ys[0].dtype, device=ys[0].device)
    _check(x, "x", (N, C, H, W), ys[0].dtype)
    _raise_on(lib.ssba_haar_iwt_pyramid(_ptr_array(ys), x.data_ptr(), N, C, H, W, levels, nb, _dtype_code(x),
                                        _stream_ptr(stream)))
    return x


def get_status() -> int:
    """ssba_get_status: read-and-clear the device status word (call after a sync)."""
    lib = load_library()
    v = ctypes.c_int32(0)
    _raise_on(lib.ssba_get_status(ctypes.byref(v)))
    return int(v.value)


def realized_sparsity(desc: SsbaDesc) -> float:
    """Dropped share of the key blocks, (Tb - keep) / Tb, with keep from ssba_keep_count
    (the library's sparsity rule; no device call)."""
    return (desc.Tb - keep_count(desc)) / desc.Tb


class BoundSelectLayer:
    """One SSBA layer on the one-launch selection path: ``pool()`` (ssba_pool_blocks) and
    ``attend()`` (ssba_forward_select, which also writes the kept-block lists), or ``fused()``
    (ssba_forward_fused: both in one launch), buffers validated once and bare C calls after
    that."""

    def __init__(self, desc: SsbaDesc, Q, K, V, qb, kb, kv_idx, kv_cnt, O, lse, stream=None,
                 fwd_workspace="default"):
        lib = load_library()
        self._lib = lib
        self._d = desc.c()
        keep = keep_count(desc)
        shp = (desc.B, desc.heads, desc.N, desc.head_dim)
        pshp = (desc.B, desc.heads, desc.Tb, desc.head_dim)
        for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O")):
            _check(t, n, shp, desc.dtype)
        _check(qb, "qb", pshp, torch.float32)
        _check(kb, "kb", pshp, torch.float32)
        _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
        _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
        _check(lse, "lse", shp[:3], torch.float32)
        if isinstance(fwd_workspace, str):
            fwd_workspace = default_forward_workspace(desc, Q.device, stream)
        fwp, fwn = _ws_args(fwd_workspace)
        if fwp is not None and fwn < forward_workspace_bytes(desc):
            raise SsbaError(SSBA_ERR_WORKSPACE, f"forward workspace needs {forward_workspace_bytes(desc)} bytes")
        self.tensors = (Q, K, V, qb, kb, kv_idx, kv_cnt, O, lse, fwd_workspace)  # keep alive
        st = _stream_ptr(stream)
        self._pool_args = (ctypes.byref(self._d), Q.data_ptr(), K.data_ptr(), qb.data_ptr(), kb.data_ptr(), st)
        self._fwd_args = (ctypes.byref(self._d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), qb.data_ptr(),
                          kb.data_ptr(), kv_idx.data_ptr(), kv_cnt.data_ptr(), None, O.data_ptr(), lse.data_ptr(),
                          fwp, fwn, st)

    def pool(self) -> None:
        rc = self._lib.ssba_pool_blocks(*self._pool_args)
        if rc:
            _raise_on(rc)

    def attend(self) -> None:
        rc = self._lib.ssba_forward_select(*self._fwd_args)
        if rc:
            _raise_on(rc)

    def fused(self) -> None:
        rc = self._lib.ssba_forward_fused(*self._fwd_args)
        if rc:
            _raise_on(rc)


class BoundLayer:
    """One SSBA layer with its buffers validated once; ``mask()`` and ``attend()`` then
    make the bare C calls (ssba_build_mask, ssba_forward) with no per-call checks, so
    that host overhead stays far below the kernels' run time in tight loops."""

    def __init__(self, desc: SsbaDesc, Q, K, V, kv_idx, kv_cnt, O, lse, workspace, stream=None,
                 fwd_workspace="default"):
        lib = load_library()
        self._lib = lib
        self._d = desc.c()
        keep = keep_count(desc)
        shp = (desc.B, desc.heads, desc.N, desc.head_dim)
        for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O")):
            _check(t, n, shp, desc.dtype)
        _check(kv_idx, "kv_idx", (desc.B, desc.heads, desc.Tb, keep), torch.int32)
        _check(kv_cnt, "kv_cnt", (desc.B, desc.heads, desc.Tb), torch.int32)
        _check(lse, "lse", shp[:3], torch.float32)
        need = mask_workspace_bytes(desc)
        if workspace.numel() * workspace.element_size() < need:
            raise SsbaError(SSBA_ERR_WORKSPACE, f"workspace needs {need} bytes")
        if isinstance(fwd_workspace, str):
            fwd_workspace = default_forward_workspace(desc, Q.device, stream) if desc.dtype == torch.bfloat16 else None
        fwp, fwn = _ws_args(fwd_workspace)
        if fwp is not None and fwn < forward_workspace_bytes(desc):
            raise SsbaError(SSBA_ERR_WORKSPACE, f"forward workspace needs {forward_workspace_bytes(desc)} bytes")
        self.tensors = (Q, K, V, kv_idx, kv_cnt, O, lse, workspace, fwd_workspace)  # keep alive
        st = _stream_ptr(stream)
        self._mask_args = (ctypes.byref(self._d), Q.data_ptr(), K.data_ptr(), kv_idx.data_ptr(),
                           kv_cnt.data_ptr(), None, workspace.data_ptr(),
                           workspace.numel() * workspace.element_size(), st)
        self._fwd_args = (ctypes.byref(self._d), Q.data_ptr(), K.data_ptr(), V.data_ptr(), kv_idx.data_ptr(),
                          kv_cnt.data_ptr(), O.data_ptr(), lse.data_ptr(), fwp, fwn, st)

    def mask(self) -> None:
        rc = self._lib.ssba_build_mask(*self._mask_args)
        if rc:
            _raise_on(rc)

    def attend(self) -> None:
        rc = self._lib.ssba_forward(*self._fwd_args)
        if rc:
            _raise_on(rc)
