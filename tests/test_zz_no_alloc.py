"""ssba_build_mask_noalloc: the mask build for callers that cannot allocate device memory
(a plug-in inside a runtime that owns all device memory, a latency-critical loop where a
cudaMalloc/cudaFree pair would synchronise the device). Its scratch is a fixed area inside
the library instead of a caller workspace, so its results must equal those of
ssba_build_mask on the same inputs, call after call, although the area keeps the previous
call's contents. This file is collected last so that a failure here cannot hide another."""
import ctypes

import pytest
import torch

from paper_2605_15684_gb300 import api, build, synthetic

FAKE = 0x100000  # aligned, never dereferenced


def test_noalloc_rejects_layers_larger_than_its_scratch():
    build.build()
    lib = api.load_library()
    big = api.SsbaDesc(B=8, heads=24, H_tok=128, W_tok=128, rho=0.84).c()  # 25 MB of scratch
    need = lib.ssba_mask_workspace_bytes(ctypes.byref(big))
    assert need > (4 << 20)
    rc = lib.ssba_build_mask_noalloc(ctypes.byref(big), FAKE, FAKE, FAKE, FAKE, None, None)
    assert rc == api.SSBA_ERR_UNSUPPORTED
    assert str(need).encode() in lib.ssba_last_error()


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    build.build()
    api.load_library()
    cases = [  # two calls in a row, different layers: 1024 px shifted, then 2048 px (largest that fits)
        (api.SsbaDesc(1, 24, 64, 64, shift_r=4, shift_c=4, rho=0.8416), 1),
        (api.SsbaDesc(1, 24, 128, 128, shift_r=4, shift_c=4, rho=0.84), 2),
        (api.SsbaDesc(1, 2, 16, 16, shift_r=3, shift_c=-5, rho=0.75, dtype=torch.float32), 3),
        (api.SsbaDesc(1, 24, 64, 64, rho=0.8416), 4),
    ]
    for desc, seed in cases:
        q, k, _ = synthetic.qkv(desc.B, desc.heads, desc.N, desc.head_dim, desc.dtype, seed=seed)
        q, k = q.cuda(), k.cuda()
        ref_idx, ref_cnt, ref_S = api.build_mask(desc, q, k, scores=True)
        idx, cnt, S = api.build_mask_noalloc(desc, q, k, scores=True)
        torch.cuda.synchronize()
        # same kernels on the same inputs: lists, counts and scores are identical
        assert torch.equal(idx, ref_idx)
        assert torch.equal(cnt, ref_cnt)
        assert torch.equal(S, ref_S)
    assert api.get_status() == api.SSBA_OK


@pytest.mark.gpu
def test_noalloc_scratch_area_on_consecutive_calls():
    """Layers that the one-launch mask kernel does not take (head_dim other than 64, or more
    than 256 blocks per row) pool into the scratch area and select from it, so these calls
    read and write the built-in area. They run back to back on different shapes, the first
    one filling almost all of the 4 MiB, so every later call finds the previous call's
    means there; each must still equal ssba_build_mask with a workspace of its own."""
    build.build()
    lib = api.load_library()
    cases = [
        # 136 x 136 grid: Tb = 289 > 256; 28 heads fill 4.14 of the 4.19 MB
        (api.SsbaDesc(1, 28, 136, 136, shift_r=4, shift_c=4, rho=0.84), 21),
        (api.SsbaDesc(1, 8, 64, 64, head_dim=128, shift_r=4, shift_c=4, rho=0.8416), 22),
        (api.SsbaDesc(1, 3, 136, 136, rho=0.9), 23),
        (api.SsbaDesc(2, 5, 24, 40, head_dim=32, shift_r=3, shift_c=-5, rho=0.6, dtype=torch.float32), 24),
        (api.SsbaDesc(1, 8, 64, 64, head_dim=128, shift_r=4, shift_c=4, rho=0.8416), 25),
    ]
    need0 = lib.ssba_mask_workspace_bytes(ctypes.byref(cases[0][0].c()))
    assert (4 << 20) - (64 << 10) < need0 <= (4 << 20)
    for desc, seed in cases:
        q, k, _ = synthetic.qkv(desc.B, desc.heads, desc.N, desc.head_dim, desc.dtype, seed=seed)
        q, k = q.cuda(), k.cuda()
        idx, cnt, S = api.build_mask_noalloc(desc, q, k, scores=True)
        ref_idx, ref_cnt, ref_S = api.build_mask(desc, q, k, scores=True)
        torch.cuda.synchronize()
        assert torch.equal(idx, ref_idx)
        assert torch.equal(cnt, ref_cnt)
        assert torch.equal(S, ref_S)
    assert api.get_status() == api.SSBA_OK
