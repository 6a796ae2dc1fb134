"""Test infrastructure: the fp64 CPU oracle for Shift Sparse Block Attention.

This package is NOT part of the product. Only ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import it. It wraps ``ssba_oracle.c``
(plain C loops in double precision, written from Sec. 2.2 and Algorithm 1 of the
paper) through ctypes and shares no code with the CUDA library.

Every function takes numpy arrays, widens them to float64 (bf16 and fp32 widen
exactly) and returns numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ssba_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libssba_oracle.so")
_lock = threading.Lock()
_lib = None

_I32P = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_F64P = np.ctypeslib.ndpointer(dtype=np.float64, flags="C_CONTIGUOUS")


def build(force: bool = False) -> str:
    """Compile ssba_oracle.c into libssba_oracle.so next to it (gcc, -O2, OpenMP)."""
    if force or not os.path.exists(_LIB_PATH) or (
        os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    ):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
               "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        c_int, c_double = ctypes.c_int, ctypes.c_double
        lib.ssba_oracle_drop_count.argtypes = [c_int, c_double]
        lib.ssba_oracle_keep_count.argtypes = [c_int, c_double]
        lib.ssba_oracle_partition.argtypes = [c_int, c_int, c_int, c_int, c_int, _I32P]
        lib.ssba_oracle_pool.argtypes = [_F64P, c_int, c_int, _I32P, c_int, _F64P]
        lib.ssba_oracle_affinity.argtypes = [_F64P, _F64P, c_int, c_int, _F64P]
        lib.ssba_oracle_gate.argtypes = [_F64P, c_int, c_int, _I32P]
        lib.ssba_oracle_attention.argtypes = [_F64P, _F64P, _F64P, c_int, c_int, _I32P, c_int,
                                              _I32P, c_int, c_double, _F64P, _F64P]
        lib.ssba_oracle_attention_rows.argtypes = [_F64P, _F64P, _F64P, c_int, c_int, _I32P, c_int,
                                                   _I32P, c_int, c_double, _I32P, c_int, _F64P, _F64P]
        lib.ssba_oracle_dense_attention.argtypes = [_F64P, _F64P, _F64P, c_int, c_int, c_double,
                                                    _F64P, _F64P]
        lib.ssba_oracle_build_mask_all.argtypes = [_F64P, _F64P, c_int, c_int, c_int, c_int, c_int,
                                                   c_int, c_int, c_double, _I32P, _I32P,
                                                   ctypes.c_void_p]
        lib.ssba_oracle_forward_all.argtypes = [_F64P, _F64P, _F64P, c_int, c_int, c_int, c_int,
                                                c_int, c_int, c_int, _I32P, c_int, c_double,
                                                _F64P, _F64P]
        lib.ssba_oracle_dense_all.argtypes = [_F64P, _F64P, _F64P, c_int, c_int, c_int, c_double,
                                              _F64P, _F64P]
        lib.ssba_oracle_attention_backward.argtypes = [_F64P, _F64P, _F64P, _F64P, c_int, c_int, _I32P, c_int,
                                                       _I32P, c_int, c_double, _F64P, _F64P, _F64P]
        lib.ssba_oracle_backward_all.argtypes = [_F64P, _F64P, _F64P, _F64P, c_int, c_int, c_int, c_int, c_int,
                                                 c_int, c_int, _I32P, c_int, c_double, _F64P, _F64P, _F64P]
        lib.ssba_oracle_haar_dwt.argtypes = [_F64P, c_int, c_int, c_int, c_int, _F64P]
        lib.ssba_oracle_haar_iwt.argtypes = [_F64P, c_int, c_int, c_int, c_int, _F64P]
        vp = ctypes.c_void_p
        lib.ssba_oracle_attention_joint.argtypes = [_F64P, _F64P, _F64P, c_int, c_int, vp, vp, c_int, _I32P,
                                                    c_int, _I32P, c_int, c_double, _F64P, _F64P]
        lib.ssba_oracle_forward_joint_all.argtypes = [_F64P, _F64P, _F64P, vp, vp, c_int, c_int, c_int, c_int,
                                                      c_int, c_int, c_int, c_int, _I32P, c_int, c_double,
                                                      _F64P, _F64P]
        lib.ssba_oracle_set_threads.argtypes = [c_int]
        lib.ssba_oracle_set_threads.restype = None
        _lib = lib
        return lib


def _f64(x) -> np.ndarray:
    if hasattr(x, "detach"):  # torch tensor: widen on the CPU, exactly
        x = x.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


def _check(rc: int, what: str) -> None:
    if rc != 0:
        raise ValueError(f"oracle: {what} rejected its arguments")


def max_threads() -> int:
    return int(_load().ssba_oracle_max_threads())


def set_threads(n: int) -> None:
    _load().ssba_oracle_set_threads(int(n))


def drop_count(Tb: int, rho: float) -> int:
    """k = floor(Tb * rho), the number of key blocks dropped per query block."""
    return int(_load().ssba_oracle_drop_count(int(Tb), float(rho)))


def keep_count(Tb: int, rho: float) -> int:
    return int(_load().ssba_oracle_keep_count(int(Tb), float(rho)))


def partition(H: int, W: int, blk: int = 8, shift=(0, 0)) -> np.ndarray:
    """Block label of every token of an H x W grid after the cyclic shift."""
    out = np.empty(H * W, dtype=np.int32)
    _check(_load().ssba_oracle_partition(H, W, blk, int(shift[0]), int(shift[1]), out),
           "partition")
    return out


def pool(X, block_of: np.ndarray, Tb: int) -> np.ndarray:
    X = _f64(X)
    N, d = X.shape
    out = np.empty((Tb, d), dtype=np.float64)
    _check(_load().ssba_oracle_pool(X, N, d, np.ascontiguousarray(block_of, np.int32), Tb, out),
           "pool")
    return out


def affinity(qb, kb) -> np.ndarray:
    qb, kb = _f64(qb), _f64(kb)
    Tb, d = qb.shape
    out = np.empty((Tb, Tb), dtype=np.float64)
    _check(_load().ssba_oracle_affinity(qb, kb, Tb, d, out), "affinity")
    return out


def gate(S, k_drop: int) -> np.ndarray:
    """Kept key-block labels per row, ascending, after dropping the k_drop smallest."""
    S = _f64(S)
    Tb = S.shape[0]
    out = np.empty((Tb, Tb - k_drop), dtype=np.int32)
    _check(_load().ssba_oracle_gate(S, Tb, int(k_drop), out), "gate")
    return out


def attention(Q, K, V, block_of, idx, scale=None):
    """Single-slice sparse attention; returns (O [N,d], lse [N])."""
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    N, d = Q.shape
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    Tb, keep = idx.shape
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((N, d), dtype=np.float64)
    lse = np.empty(N, dtype=np.float64)
    _check(_load().ssba_oracle_attention(Q, K, V, N, d, np.ascontiguousarray(block_of, np.int32),
                                         Tb, idx, keep, scale, O, lse), "attention")
    return O, lse


def attention_rows(Q, K, V, block_of, idx, rows, scale=None):
    """Single-slice sparse attention for the listed query tokens only."""
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    N, d = Q.shape
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    Tb, keep = idx.shape
    rows = np.ascontiguousarray(rows, dtype=np.int32)
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((rows.shape[0], d), dtype=np.float64)
    lse = np.empty(rows.shape[0], dtype=np.float64)
    _check(_load().ssba_oracle_attention_rows(Q, K, V, N, d, np.ascontiguousarray(block_of, np.int32),
                                              Tb, idx, keep, scale, rows, rows.shape[0], O, lse),
           "attention_rows")
    return O, lse


def dense_attention(Q, K, V, scale=None):
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    N, d = Q.shape
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((N, d), dtype=np.float64)
    lse = np.empty(N, dtype=np.float64)
    _check(_load().ssba_oracle_dense_attention(Q, K, V, N, d, scale, O, lse), "dense_attention")
    return O, lse


def build_mask(Q, K, H: int, W: int, blk: int = 8, shift=(0, 0), rho: float = 0.0,
               return_scores: bool = False):
    """Whole-tensor mask build. Q, K: [B, heads, N, d]. Returns (idx, cnt[, S])."""
    Q, K = _f64(Q), _f64(K)
    B, h, N, d = Q.shape
    if N != H * W:
        raise ValueError("N must equal H*W")
    Tb = N // (blk * blk)
    keep = keep_count(Tb, rho)
    idx = np.empty((B, h, Tb, keep), dtype=np.int32)
    cnt = np.empty((B, h, Tb), dtype=np.int32)
    S = np.empty((B, h, Tb, Tb), dtype=np.float64) if return_scores else None
    _check(_load().ssba_oracle_build_mask_all(
        Q, K, B * h, H, W, d, blk, int(shift[0]), int(shift[1]), float(rho), idx, cnt,
        S.ctypes.data if S is not None else None), "build_mask")
    return (idx, cnt, S) if return_scores else (idx, cnt)


def forward(Q, K, V, idx, H: int, W: int, blk: int = 8, shift=(0, 0), scale=None):
    """Whole-tensor sparse forward. Q, K, V: [B, heads, N, d]; idx [B, heads, Tb, keep]."""
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    B, h, N, d = Q.shape
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    keep = idx.shape[-1]
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((B, h, N, d), dtype=np.float64)
    lse = np.empty((B, h, N), dtype=np.float64)
    _check(_load().ssba_oracle_forward_all(Q, K, V, B * h, H, W, d, blk, int(shift[0]),
                                           int(shift[1]), idx, keep, scale, O, lse), "forward")
    return O, lse


def attention_joint(Q, K, V, Kt, Vt, block_of, idx, scale=None):
    """Single-slice joint text + image attention (Algorithm 1 with its text segment):
    Q, K, V [N, d] image tokens, Kt, Vt [Tt, d] text tokens; returns the image rows
    (O [N, d], lse [N])."""
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    N, d = Q.shape
    Kt, Vt = _f64(Kt).reshape(-1, d), _f64(Vt).reshape(-1, d)
    Tt = Kt.shape[0]
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    Tb, keep = idx.shape
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((N, d), dtype=np.float64)
    lse = np.empty(N, dtype=np.float64)
    _check(_load().ssba_oracle_attention_joint(Q, K, V, N, d, Kt.ctypes.data if Tt else None,
                                               Vt.ctypes.data if Tt else None, Tt,
                                               np.ascontiguousarray(block_of, np.int32), Tb, idx, keep, scale,
                                               O, lse), "attention_joint")
    return O, lse


def forward_joint(Q, K, V, Kt, Vt, idx, H: int, W: int, blk: int = 8, shift=(0, 0), scale=None):
    """Whole-tensor joint forward. Q, K, V: [B, heads, N, d]; Kt, Vt: [B, heads, Tt, d];
    idx [B, heads, Tb, keep]. Returns the image rows (O [B, heads, N, d], lse)."""
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    Kt, Vt = _f64(Kt), _f64(Vt)
    B, h, N, d = Q.shape
    Tt = Kt.shape[2]
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    keep = idx.shape[-1]
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((B, h, N, d), dtype=np.float64)
    lse = np.empty((B, h, N), dtype=np.float64)
    _check(_load().ssba_oracle_forward_joint_all(Q, K, V, Kt.ctypes.data if Tt else None,
                                                 Vt.ctypes.data if Tt else None, Tt, B * h, H, W, d, blk,
                                                 int(shift[0]), int(shift[1]), idx, keep, scale, O, lse),
           "forward_joint")
    return O, lse


def attention_backward(Q, K, V, dO, block_of, idx, scale=None):
    """Single-slice gradients (dQ, dK, dV) of the sparse attention for output gradient dO."""
    Q, K, V, dO = _f64(Q), _f64(K), _f64(V), _f64(dO)
    N, d = Q.shape
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    Tb, keep = idx.shape
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    dQ, dK, dV = (np.empty((N, d), dtype=np.float64) for _ in range(3))
    _check(_load().ssba_oracle_attention_backward(Q, K, V, dO, N, d, np.ascontiguousarray(block_of, np.int32),
                                                  Tb, idx, keep, scale, dQ, dK, dV), "attention_backward")
    return dQ, dK, dV


def backward(Q, K, V, dO, idx, H: int, W: int, blk: int = 8, shift=(0, 0), scale=None):
    """Whole-tensor gradients of the sparse forward. Q, K, V, dO: [B, heads, N, d]."""
    Q, K, V, dO = _f64(Q), _f64(K), _f64(V), _f64(dO)
    B, h, N, d = Q.shape
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    keep = idx.shape[-1]
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    dQ, dK, dV = (np.empty((B, h, N, d), dtype=np.float64) for _ in range(3))
    _check(_load().ssba_oracle_backward_all(Q, K, V, dO, B * h, H, W, d, blk, int(shift[0]), int(shift[1]), idx,
                                            keep, scale, dQ, dK, dV), "backward")
    return dQ, dK, dV


def dense_forward(Q, K, V, scale=None):
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    B, h, N, d = Q.shape
    scale = 1.0 / np.sqrt(d) if scale is None else float(scale)
    O = np.empty((B, h, N, d), dtype=np.float64)
    lse = np.empty((B, h, N), dtype=np.float64)
    _check(_load().ssba_oracle_dense_all(Q, K, V, B * h, N, d, scale, O, lse), "dense_forward")
    return O, lse


def haar_dwt(x, nb: int = 4):
    """One Haar level per channel: x [..., C, H, W] -> [..., nb * C, H/2, W/2] (LL, HL, LH, HH)."""
    x = _f64(x)
    *lead, C, H, W = x.shape
    xs = x.reshape(-1, C, H, W)
    y = np.empty((xs.shape[0], nb * C, H // 2, W // 2), dtype=np.float64)
    for i in range(xs.shape[0]):
        _check(_load().ssba_oracle_haar_dwt(np.ascontiguousarray(xs[i]), C, H, W, nb, y[i]), "haar_dwt")
    return y.reshape(*lead, nb * C, H // 2, W // 2)


def haar_iwt(y, C: int, nb: int = 4):
    """Inverse Haar level: y [..., nb * C, h, w] -> [..., C, 2h, 2w] (HH = 0 when nb = 3)."""
    y = _f64(y)
    *lead, nbC, h, w = y.shape
    ys = y.reshape(-1, nbC, h, w)
    x = np.empty((ys.shape[0], C, 2 * h, 2 * w), dtype=np.float64)
    for i in range(ys.shape[0]):
        _check(_load().ssba_oracle_haar_iwt(np.ascontiguousarray(ys[i]), C, 2 * h, 2 * w, nb, x[i]), "haar_iwt")
    return x.reshape(*lead, C, 2 * h, 2 * w)


def haar_dwt_pyramid(x, levels: int, nb: int = 4):
    """The encoder's recursion (Sec. 2.3, Eq. for W^(l)) without the convolutions between
    levels: level 1 is the bank applied to x, level l the bank applied to the LL band of level
    l - 1. Returns [W^(1), ..., W^(levels)], W^(l) [..., nb * C, H / 2^l, W / 2^l]."""
    x = _f64(x)
    C = x.shape[-3]
    out, cur = [], x
    for _ in range(levels):
        y = haar_dwt(cur, nb)
        out.append(y)
        cur = y[..., :C, :, :]  # the LL band of every channel
    return out


def haar_iwt_pyramid(ys, C: int, nb: int = 4):
    """The decoder's inverse pyramid (Sec. 2.3) without the refinements between levels: the
    deepest level is inverted whole, and each shallower level is inverted with its LL band
    replaced by the level below's reconstruction. Only LL of the deepest level and the detail
    bands are read. Returns x [..., C, H, W]."""
    cur = None
    for y in reversed([_f64(t) for t in ys]):
        if cur is not None:
            y = y.copy()
            y[..., :C, :, :] = cur
        cur = haar_iwt(y, C, nb)
    return cur


ROPE_BASE = 10000.0


def rope_2d(x, H: int, W: int, base: float = ROPE_BASE):
    """Rotary position embedding of image tokens (Algorithm 1, first step), 2-D axial
    reading: x [..., N, d] with N = H*W tokens in row-major grid order; the first d/2
    dimensions rotate with the token's row r, the last d/2 with its column c. Within each
    half, the pair (2i, 2i+1) turns by pos * theta_i, theta_i = base^(-i / (d/4))."""
    x = _f64(x)
    N, d = x.shape[-2], x.shape[-1]
    if N != H * W or d % 4:
        raise ValueError("rope_2d: N must equal H*W and d be a multiple of 4")
    half, nf = d // 2, d // 4
    theta = base ** (-np.arange(nf, dtype=np.float64) / nf)
    n = np.arange(N)
    out = x.copy()
    for off, pos in ((0, n // W), (half, n % W)):
        ang = pos[:, None].astype(np.float64) * theta[None, :]
        cos, sin = np.cos(ang), np.sin(ang)
        even = x[..., off:off + half:2]
        odd = x[..., off + 1:off + half:2]
        out[..., off:off + half:2] = even * cos - odd * sin
        out[..., off + 1:off + half:2] = even * sin + odd * cos
    return out


def qkv_rope(X, Wqkv, bias, heads: int, H: int, W: int, d: int = 64):
    """The QKV projection and RoPE that precede the mask build (Algorithm 1): X [B, N, Dm],
    Wqkv [3 * heads * d, Dm] (rows: Q heads, then K heads, then V heads), bias [3 * heads * d]
    or None. Returns Q, K, V [B, heads, N, d] with RoPE applied to Q and K."""
    X, Wqkv = _f64(X), _f64(Wqkv)
    B, N, Dm = X.shape
    Y = X @ Wqkv.T
    if bias is not None:
        Y = Y + _f64(bias)
    Y = Y.reshape(B, N, 3, heads, d).transpose(2, 0, 3, 1, 4)  # [3, B, heads, N, d]
    return rope_2d(Y[0], H, W), rope_2d(Y[1], H, W), np.ascontiguousarray(Y[2])


def pooled_blocks(X, H: int, W: int, blk: int = 8, shift=(0, 0)):
    """Block means of every (batch, head): X [B, heads, N, d] -> [B, heads, Tb, d]."""
    X = _f64(X)
    B, h, N, d = X.shape
    lab = partition(H, W, blk, shift)
    Tb = N // (blk * blk)
    out = np.empty((B, h, Tb, d), dtype=np.float64)
    for b in range(B):
        for i in range(h):
            out[b, i] = pool(X[b, i], lab, Tb)
    return out
