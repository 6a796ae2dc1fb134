"""Host-side checks of the C-ABI library: it builds, loads without a GPU, exports
every symbol include/ssba.h declares, and its host validation returns the
documented status codes before any device work (no compute call is made here)."""
import ctypes
import math
import os
import re
import subprocess

import pytest

import oracle
from paper_2605_15684_gb300 import api, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ssba.h")
FAKE = 0x100000  # a 16-byte aligned, never dereferenced address


@pytest.fixture(scope="module")
def lib():
    build.build()
    return api.load_library()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"SSBA_API\s+[\w\s\*]+?\b(ssba_\w+)\s*\(", text)))


def desc(**kw):
    base = dict(B=1, heads=2, H_tok=16, W_tok=16, head_dim=64, block=8, shift_r=4, shift_c=4, rho=0.75,
                dtype=api.SSBA_BF16, softmax_scale=0.0)
    base.update(kw)
    return api._Desc(**base)


def test_header_declares_the_documented_entry_points():
    assert declared_symbols() == sorted(api.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", api.library_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (ssba_\w+)", out))
    assert set(declared_symbols()) <= exported
    # nothing else of ours leaks out of the library
    assert exported == set(declared_symbols())


@pytest.mark.parametrize("H,W,rho", [(16, 16, 0.75), (32, 32, 0.8416), (64, 64, 0.8416), (64, 64, 0.85),
                                     (128, 128, 0.84), (128, 128, 0.9), (16, 40, 0.5), (64, 64, 0.0)])
def test_keep_count_matches_the_sparsity_rule(lib, H, W, rho):
    Tb = H * W // 64
    d = desc(H_tok=H, W_tok=W, rho=rho)
    assert lib.ssba_keep_count(ctypes.byref(d)) == Tb - math.floor(Tb * rho) == oracle.keep_count(Tb, rho)


def test_workspace_bytes(lib):
    d = desc(B=1, heads=24, H_tok=64, W_tok=64)
    one = 24 * 64 * 64 * 4
    assert lib.ssba_mask_workspace_bytes(ctypes.byref(d)) == 2 * ((one + 255) // 256 * 256)
    assert lib.ssba_mask_workspace_bytes(ctypes.byref(desc(H_tok=12))) == 0


@pytest.mark.parametrize("bad", [dict(H_tok=12), dict(W_tok=0), dict(rho=1.0), dict(rho=-0.1),
                                 dict(dtype=7), dict(B=0), dict(softmax_scale=-1.0),
                                 dict(head_dim=0)])
def test_invalid_descriptors_are_rejected(lib, bad):
    d = desc(**bad)
    assert lib.ssba_keep_count(ctypes.byref(d)) == -1
    rc = lib.ssba_forward(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, 0, None)
    assert rc == api.SSBA_ERR_INVALID
    assert lib.ssba_last_error()


def test_null_and_misaligned_pointers(lib):
    d = desc()
    ws = lib.ssba_mask_workspace_bytes(ctypes.byref(d))
    assert lib.ssba_build_mask(ctypes.byref(d), None, FAKE, FAKE, FAKE, None, FAKE, ws, None) == \
        api.SSBA_ERR_INVALID
    assert lib.ssba_build_mask(ctypes.byref(d), FAKE + 2, FAKE, FAKE, FAKE, None, FAKE, ws, None) == \
        api.SSBA_ERR_INVALID
    assert lib.ssba_build_mask(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, None, FAKE, ws - 1, None) == \
        api.SSBA_ERR_WORKSPACE
    assert lib.ssba_build_mask(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, None, None, ws, None) == \
        api.SSBA_ERR_WORKSPACE
    assert lib.ssba_forward(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, None, 0, None) == \
        api.SSBA_ERR_INVALID
    assert lib.ssba_forward(ctypes.byref(d), FAKE, FAKE, FAKE + 8, FAKE, FAKE, FAKE, FAKE, None, 0, None) == \
        api.SSBA_ERR_INVALID
    assert b"aligned" in lib.ssba_last_error()


@pytest.mark.parametrize("bad", [dict(shift_r=2), dict(shift_c=-6), dict(head_dim=128), dict(block=16, H_tok=32,
                                                                                            W_tok=32)])
def test_tensor_core_path_rejects_unsupported_shapes(lib, bad):
    """The bf16 path needs head_dim 64, 8x8 blocks and 4-aligned shifts; it says so before launching."""
    d = desc(**bad)
    rc = lib.ssba_forward(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, 0, None)
    assert rc == api.SSBA_ERR_UNSUPPORTED
    assert b"multiples of 4" in lib.ssba_last_error()


def test_forward_workspace_rules(lib):
    """The optional forward workspace: sized by the library, checked for size and
    alignment before any launch, and not needed by the fp32 path."""
    d = desc()
    need = lib.ssba_forward_workspace_bytes(ctypes.byref(d))
    assert need > 0 and need % 16 == 0
    assert lib.ssba_forward_workspace_bytes(ctypes.byref(desc(dtype=api.SSBA_FP32))) == 0
    assert lib.ssba_forward_workspace_bytes(ctypes.byref(desc(H_tok=12))) == 0
    args = (ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE)
    assert lib.ssba_forward(*args, FAKE, need - 16, None) == api.SSBA_ERR_WORKSPACE
    assert b"workspace" in lib.ssba_last_error()
    assert lib.ssba_forward(*args, FAKE + 8, need, None) == api.SSBA_ERR_INVALID
    assert lib.ssba_forward_dense(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 16, None) == \
        api.SSBA_ERR_WORKSPACE


def test_forward_joint_validation(lib):
    """The joint text + image entry point checks its text arguments before any launch."""
    d = desc()
    base = (FAKE, FAKE, FAKE)
    tail = (FAKE, FAKE, FAKE, FAKE, None, 0, None)
    assert lib.ssba_forward_joint(ctypes.byref(d), *base, None, None, 16, *tail) == api.SSBA_ERR_INVALID
    assert lib.ssba_forward_joint(ctypes.byref(d), *base, FAKE, FAKE, -1, *tail) == api.SSBA_ERR_INVALID
    assert lib.ssba_forward_joint(ctypes.byref(d), *base, FAKE + 8, FAKE, 16, *tail) == api.SSBA_ERR_INVALID
    assert lib.ssba_forward_joint(ctypes.byref(desc(dtype=api.SSBA_FP32)), *base, FAKE, FAKE, 16, *tail) == \
        api.SSBA_ERR_UNSUPPORTED
    assert b"bf16" in lib.ssba_last_error()


def test_backward_validation(lib):
    """The backward entry point checks its workspace and shape before any launch."""
    d = desc()
    need = lib.ssba_backward_workspace_bytes(ctypes.byref(d))
    # D per row, a 256-byte counter, the transposed lists (offsets, counts, entries), then the
    # rows' (lse, D) pairs by block, each part rounded up to 256 bytes
    up = lambda x: (x + 255) // 256 * 256
    BH, N, Tb, keep = 1 * 2, 16 * 16, 4, lib.ssba_keep_count(ctypes.byref(d))
    assert need == up(BH * N * 4) + 256 + 2 * up(BH * Tb * 4) + up(BH * Tb * keep * 4) + up(BH * N * 8)
    args = [ctypes.byref(d)] + [FAKE] * 11
    assert lib.ssba_backward(*args, FAKE, need - 4, None) == api.SSBA_ERR_WORKSPACE
    assert lib.ssba_backward(*args, None, need, None) == api.SSBA_ERR_WORKSPACE
    bad = [ctypes.byref(d)] + [FAKE] * 5 + [None] + [FAKE] * 5
    assert lib.ssba_backward(*bad, FAKE, need, None) == api.SSBA_ERR_INVALID
    for i in (1, 2, 3, 4, 6, 9, 10, 11):  # Q, K, V, O, dO, dQ, dK, dV: 16-byte aligned or rejected
        mis = list(args)
        mis[i] = FAKE + 4
        assert lib.ssba_backward(*mis, FAKE, need, None) == api.SSBA_ERR_INVALID, i
    assert b"16-byte" in lib.ssba_last_error()
    assert lib.ssba_backward_workspace_bytes(ctypes.byref(desc(H_tok=12))) == 0


def test_haar_validation(lib):
    """The Haar entry points check sizes, band count, dtype and alignment before any launch."""
    ok = (1, 3, 8, 8, 4, api.SSBA_FP32, None)
    for fn in (lib.ssba_haar_dwt, lib.ssba_haar_iwt):
        assert fn(FAKE, FAKE, 1, 3, 7, 8, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # odd H
        assert fn(FAKE, FAKE, 1, 3, 8, 9, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # odd W
        assert fn(FAKE, FAKE, 1, 3, 8, 8, 2, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # nb not 3 or 4
        assert fn(FAKE, FAKE, 0, 3, 8, 8, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # empty batch
        assert fn(FAKE, FAKE, 1, 3, 8, 8, 4, 7, None) == api.SSBA_ERR_INVALID  # unknown dtype
        assert fn(None, FAKE, *ok) == api.SSBA_ERR_INVALID
        assert fn(FAKE + 4, FAKE, *ok) == api.SSBA_ERR_INVALID  # misaligned input
        assert fn(FAKE, FAKE + 8, *ok) == api.SSBA_ERR_INVALID  # misaligned output
    assert b"ssba_haar_iwt" in lib.ssba_last_error()


def test_haar_pyramid_validation(lib):
    """Level count, divisibility by 2^levels and every level's pointer are checked first."""
    import ctypes as ct
    ys = (ct.c_void_p * 3)(FAKE, FAKE, FAKE)
    for fn, first in ((lib.ssba_haar_dwt_pyramid, (FAKE, ys)), (lib.ssba_haar_iwt_pyramid, (ys, FAKE))):
        assert fn(*first, 1, 2, 16, 16, 4, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # 4 levels
        assert fn(*first, 1, 2, 16, 16, 0, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # 0 levels
        assert fn(*first, 1, 2, 12, 16, 3, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # 12 % 8
        assert fn(*first, 1, 2, 16, 20, 3, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID  # 20 % 8
    bad = (ct.c_void_p * 3)(FAKE, FAKE + 4, FAKE)
    assert lib.ssba_haar_dwt_pyramid(FAKE, bad, 1, 2, 16, 16, 3, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID
    assert lib.ssba_haar_dwt_pyramid(FAKE, None, 1, 2, 16, 16, 3, 4, api.SSBA_FP32, None) == api.SSBA_ERR_INVALID
    assert b"ssba_haar_dwt_pyramid" in lib.ssba_last_error()


def test_qkv_and_select_validation(lib):
    """The fused projection and the selection check pointers, pairing and shape first."""
    d = desc()
    good = [FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE]  # X W bias Q K V qb kb
    args = lambda v: [ct_byref(d)] + v + [None]
    bad = list(good)
    bad[6] = None  # qb without kb
    assert lib.ssba_qkv_rope_pool(*args(bad)) == api.SSBA_ERR_INVALID
    bad = list(good)
    bad[0] = None
    assert lib.ssba_qkv_rope_pool(*args(bad)) == api.SSBA_ERR_INVALID
    bad = list(good)
    bad[3] = FAKE + 8
    assert lib.ssba_qkv_rope_pool(*args(bad)) == api.SSBA_ERR_INVALID
    d32 = desc(dtype=api.SSBA_FP32)
    assert lib.ssba_qkv_rope_pool(ct_byref(d32), *good, None) == api.SSBA_ERR_UNSUPPORTED
    dsh = desc(shift_r=3)
    assert lib.ssba_qkv_rope_pool(ct_byref(dsh), *good, None) == api.SSBA_ERR_UNSUPPORTED
    assert b"multiples of 4" in lib.ssba_last_error()
    assert lib.ssba_select_mask(ct_byref(d), None, FAKE, FAKE, FAKE, None, None) == api.SSBA_ERR_INVALID
    assert lib.ssba_select_mask(ct_byref(d), FAKE + 4, FAKE, FAKE, FAKE, None, None) == api.SSBA_ERR_INVALID
    assert lib.ssba_select_mask(ct_byref(desc(head_dim=66)), FAKE, FAKE, FAKE, FAKE, None, None) == \
        api.SSBA_ERR_UNSUPPORTED


def test_pool_and_select_forward_validation(lib):
    """ssba_pool_blocks and ssba_forward_select check pointers, alignment, dtype and the row
    length before any launch."""
    d = desc()
    assert lib.ssba_pool_blocks(ctypes.byref(d), FAKE, None, FAKE, FAKE, None) == api.SSBA_ERR_INVALID
    assert lib.ssba_pool_blocks(ctypes.byref(d), FAKE, FAKE, FAKE + 4, FAKE, None) == api.SSBA_ERR_INVALID
    assert lib.ssba_pool_blocks(ctypes.byref(desc(head_dim=12)), FAKE, FAKE, FAKE, FAKE, None) == \
        api.SSBA_ERR_UNSUPPORTED
    good = [FAKE] * 11  # Q K V qb kb idx cnt scores O lse workspace
    fs = lambda dd, v, n=0: lib.ssba_forward_select(ctypes.byref(dd), *v, n, None)
    bad = list(good)
    bad[3] = None  # no block means
    assert fs(d, bad) == api.SSBA_ERR_INVALID
    bad = list(good)
    bad[8] = FAKE + 8  # misaligned O
    assert fs(d, bad) == api.SSBA_ERR_INVALID
    assert fs(desc(dtype=api.SSBA_FP32), good) == api.SSBA_ERR_UNSUPPORTED
    assert b"bf16" in lib.ssba_last_error()
    # rows longer than 256 blocks: the two-launch path
    assert fs(desc(H_tok=136, W_tok=136), good) == api.SSBA_ERR_UNSUPPORTED
    assert b"Tb <= 256" in lib.ssba_last_error()
    # the fused launch: the same checks, and a workspace is required (it holds the barrier)
    ff = lambda dd, v, n=0: lib.ssba_forward_fused(ctypes.byref(dd), *v, n, None)
    bad = list(good)
    bad[10] = None
    assert ff(d, bad) == api.SSBA_ERR_WORKSPACE
    assert b"workspace" in lib.ssba_last_error()
    bad = list(good)
    bad[4] = FAKE + 4  # misaligned kb
    assert ff(d, bad) == api.SSBA_ERR_INVALID
    assert ff(desc(dtype=api.SSBA_FP32), good) == api.SSBA_ERR_UNSUPPORTED
    assert ff(desc(H_tok=136, W_tok=136), good) == api.SSBA_ERR_UNSUPPORTED
    assert b"Tb <= 256" in lib.ssba_last_error()
    # its failure-detection hook: the same checks before any launch (workspace required)
    ft = lambda dd, v: lib.ssba_test_fused_timeout(ctypes.byref(dd), *v[:3], *v[3:5], *v[5:7], *v[8:11], 0,
                                                   2_000_000, None)
    assert ft(d, [FAKE] * 7 + [None] + [FAKE] * 2 + [None]) == api.SSBA_ERR_INVALID  # no workspace
    assert ft(desc(dtype=api.SSBA_FP32), good) == api.SSBA_ERR_UNSUPPORTED


def ct_byref(d):
    return ctypes.byref(d)


def test_build_mask_rejects_unsupported_head_dim(lib):
    d = desc(head_dim=12)  # 24 bytes per bf16 row: not a multiple of 16
    ws = lib.ssba_mask_workspace_bytes(ctypes.byref(d))
    assert lib.ssba_build_mask(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, None, FAKE, ws, None) == \
        api.SSBA_ERR_UNSUPPORTED


def test_python_binding_validates_before_calling(lib):
    import torch
    dsc = api.SsbaDesc(B=1, heads=2, H_tok=16, W_tok=16, rho=0.75)
    q = torch.zeros(1, 2, 256, 64, dtype=torch.bfloat16)
    with pytest.raises(api.SsbaError, match="CUDA tensor"):
        api.build_mask(dsc, q, q)
    with pytest.raises(api.SsbaError, match="CUDA tensor"):
        api.forward_fused(dsc, q, q, q)
    with pytest.raises(api.SsbaError, match="workspace"):
        api.forward_fused(dsc, q, q, q, workspace=None)
    assert api.realized_sparsity(api.SsbaDesc(1, 24, 64, 64, rho=0.8416)) == 53 / 64
