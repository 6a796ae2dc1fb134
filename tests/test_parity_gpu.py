"""GPU parity: the CUDA path through the C-ABI against the fp64 oracle, element by
element, on the seeded synthetic workloads (tolerances in tests/parity.py)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_15684_gb300 import api, build, synthetic
from tests.parity import check_mask, check_out

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    api.load_library()
    yield
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK


def _inputs(B, h, H, W, dtype, seed=0, std=1.0):
    q, k, v = synthetic.qkv(B, h, H * W, 64, dtype, seed, std)
    return q, k, v, q.cuda(), k.cuda(), v.cuda()


def _mask_case(B, h, H, W, dtype, shift, rho, seed=0, std=1.0):
    q, k, v, qd, kd, vd = _inputs(B, h, H, W, dtype, seed, std)
    desc = api.SsbaDesc(B, h, H, W, shift_r=shift[0], shift_c=shift[1], rho=rho, dtype=dtype)
    idx, cnt, S = api.build_mask(desc, qd, kd, scores=True)
    torch.cuda.synchronize()
    idx_o, cnt_o, S_o = oracle.build_mask(q, k, H, W, 8, shift, rho, return_scores=True)
    keep = oracle.keep_count(H * W // 64, rho)
    near = check_mask(idx.cpu().numpy(), cnt.cpu().numpy(), S.cpu().numpy(), S_o, idx_o, keep)
    return desc, (q, k, v, qd, kd, vd), idx_o, near


# ----------------------------------------------------------------------------- mask (K1)
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (-4, -4), (3, -5)])
def test_mask_tiny(dtype, shift):
    """Tiny case: 16x16 grid, 2 heads, 4 blocks, ~75% sparsity."""
    _mask_case(1, 2, 16, 16, dtype, shift, 0.75)


@pytest.mark.parametrize("H,W,B,rho,shift", [
    (32, 32, 1, 0.8416, (0, 0)),      # 512 px, unshifted layer
    (32, 32, 1, 0.8416, (4, 4)),      # 512 px, shifted layer
    (64, 64, 1, 0.8416, (4, 4)),      # 1024 px headline
    (64, 64, 4, 0.5, (0, 0)),         # elastic sweep, batch 4
    (24, 40, 2, 0.6, (4, -4)),        # non-square, odd block count (15)
    (128, 128, 1, 0.84, (4, 4)),      # 2048 px stress (Tb = 256, two key chunks)
])
def test_mask_full_configs(H, W, B, rho, shift):
    std = 0.125 if H == 32 else 1.0
    _, _, _, near = _mask_case(B, 24, H, W, torch.bfloat16, shift, rho, std=std)
    assert near < 0.1 * B * 24 * (H * W // 64)


@pytest.mark.parametrize("d,H,W,dtype", [(32, 32, 32, torch.bfloat16), (128, 32, 32, torch.float32),
                                         (64, 136, 136, torch.bfloat16)])
def test_mask_two_kernel_path(d, H, W, dtype):
    """Shapes outside the fused one-launch build (head_dim 64, at most 256 blocks) go
    through the separate pooling and selection kernels: other head widths, and 289
    blocks (radix selection)."""
    q, k, _ = synthetic.qkv(1, 2, H * W, d, dtype, 7)
    desc = api.SsbaDesc(1, 2, H, W, head_dim=d, shift_r=4, shift_c=4, rho=0.8, dtype=dtype)
    idx, cnt, S = api.build_mask(desc, q.cuda(), k.cuda(), scores=True)
    torch.cuda.synchronize()
    idx_o, cnt_o, S_o = oracle.build_mask(q, k, H, W, 8, (4, 4), 0.8, return_scores=True)
    keep = oracle.keep_count(H * W // 64, 0.8)
    near = check_mask(idx.cpu().numpy(), cnt.cpu().numpy(), S.cpu().numpy(), S_o, idx_o, keep)
    assert near < 0.1 * 2 * (H * W // 64)


def test_mask_ties_keep_lower_label():
    """Constant Q/K make every S entry equal: each row keeps labels 0..keep-1."""
    H = W = 32
    q = torch.ones(1, 2, H * W, 64, dtype=torch.bfloat16, device="cuda")
    desc = api.SsbaDesc(1, 2, H, W, shift_r=4, shift_c=4, rho=0.75)
    idx, cnt = api.build_mask(desc, q, q)
    keep = 16 - 12
    assert idx.shape == (1, 2, 16, keep)
    assert bool((idx.cpu() == torch.arange(keep, dtype=torch.int32)).all())
    assert bool((cnt.cpu() == keep).all())


def test_mask_keep_one_and_all():
    for rho, keep in ((0.95, 1), (0.0, 16)):
        desc, _, idx_o, _ = _mask_case(1, 3, 32, 32, torch.bfloat16, (4, 4), rho)
        assert idx_o.shape[-1] == keep


# ----------------------------------------------------------------------------- forward (K2/K3)
@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (3, -5)])
@pytest.mark.parametrize("rho", [0.75, 0.0])
def test_forward_fp32_tiny(shift, rho):
    """fp32 tiny case (CUDA-core kernel): <= 1e-4 against the oracle; rho = 0 is dense."""
    H = W = 16
    q, k, v, qd, kd, vd = _inputs(1, 2, H, W, torch.float32)
    desc = api.SsbaDesc(1, 2, H, W, shift_r=shift[0], shift_c=shift[1], rho=rho, dtype=torch.float32)
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, shift, rho)
    O, lse = api.forward(desc, qd, kd, vd, torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda())
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward(q, k, v, idx_o, H, W, 8, shift)
    check_out(O.cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "fp32")
    if rho == 0.0:
        O_d, lse_d = oracle.dense_forward(q, k, v)
        check_out(O.cpu().numpy(), lse.cpu().numpy(), O_d, lse_d, "fp32")


def _bf16_forward_case(B, h, H, W, shift, rho, std=1.0, seed=0):
    q, k, v, qd, kd, vd = _inputs(B, h, H, W, torch.bfloat16, seed, std)
    desc = api.SsbaDesc(B, h, H, W, shift_r=shift[0], shift_c=shift[1], rho=rho)
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, shift, rho)
    O, lse = api.forward(desc, qd, kd, vd, torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda())
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward(q, k, v, idx_o, H, W, 8, shift)
    return check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (-4, -4), (4, -8)])
def test_forward_bf16_tiny_grid(shift):
    _bf16_forward_case(1, 2, 16, 16, shift, 0.75)


@pytest.mark.parametrize("H,W,B,h,rho,shift,std", [
    (32, 32, 1, 24, 0.8416, (4, 4), 0.125),   # 512 px config (scaled inputs)
    (32, 32, 1, 24, 0.8416, (0, 0), 1.0),     # 512 px grid, unit variance
    (64, 64, 1, 24, 0.8416, (4, 4), 1.0),     # 1024 px headline (1536 items, ragged over the grid)
    (64, 64, 1, 8, 0.0, (0, 0), 1.0),         # keep = Tb: dense through the sparse kernel
    (32, 32, 2, 6, 0.95, (4, 4), 1.0),        # keep = 1
    (24, 40, 2, 5, 0.6, (4, -4), 1.0),        # non-square grid, odd Tb
])
def test_forward_bf16_configs(H, W, B, h, rho, shift, std):
    _bf16_forward_case(B, h, H, W, shift, rho, std)


def test_forward_bf16_large_logits_rescale_path():
    """Inputs scaled so that scores span tens of units: the running max must grow
    mid-row, exercising the in-TMEM O rescale."""
    H = W = 32
    q, k, v, qd, kd, vd = _inputs(1, 4, H, W, torch.float32, seed=3)
    ramp = torch.linspace(0.2, 4.0, H * W).view(1, 1, H * W, 1)
    q = (q * 3.0).to(torch.bfloat16)
    k = (k * ramp).to(torch.bfloat16)
    v = v.to(torch.bfloat16)
    desc = api.SsbaDesc(1, 4, H, W, rho=0.5)
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, (0, 0), 0.5)
    O, lse = api.forward(desc, q.cuda(), k.cuda(), v.cuda(), torch.from_numpy(idx_o).cuda(),
                         torch.from_numpy(cnt_o).cuda())
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward(q, k, v, idx_o, H, W, 8, (0, 0))
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


def test_forward_bf16_2048px_sampled_rows():
    """Full 2048 px size (N=16384, 24 heads, keep 41): GPU mask on every head against the
    oracle, GPU forward checked on sampled query rows of two heads."""
    H = W = 128
    desc, (q, k, v, qd, kd, vd), idx_o, _ = _mask_case(1, 24, H, W, torch.bfloat16, (4, 4), 0.84)
    O, lse = api.forward(desc, qd, kd, vd, torch.from_numpy(idx_o).cuda(),
                         torch.full((1, 24, 256), idx_o.shape[-1], dtype=torch.int32, device="cuda"))
    torch.cuda.synchronize()
    lab = oracle.partition(H, W, 8, (4, 4))
    rng = np.random.default_rng(0)
    rows = np.sort(rng.choice(H * W, 96, replace=False)).astype(np.int32)
    for head in (0, 23):
        O_o, lse_o = oracle.attention_rows(q[0, head], k[0, head], v[0, head], lab, idx_o[0, head], rows)
        check_out(O[0, head].float().cpu().numpy()[rows], lse[0, head].cpu().numpy()[rows], O_o, lse_o, "bf16")


def test_forward_dense_bf16():
    H = W = 32
    q, k, v, qd, kd, vd = _inputs(1, 4, H, W, torch.bfloat16)
    desc = api.SsbaDesc(1, 4, H, W)
    O, lse = api.forward_dense(desc, qd, kd, vd)
    torch.cuda.synchronize()
    O_o, lse_o = oracle.dense_forward(q, k, v)
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


@pytest.mark.parametrize("B,h,H,W", [
    (1, 24, 64, 64),   # 1024 px: the 128-token-tile kernel, 32 key tiles a row
    (2, 16, 32, 32),   # B > 1, units spread over the streams unevenly
    (1, 3, 24, 40),    # N = 960, not a multiple of 128: the 64-row path
])
def test_forward_dense_bf16_shapes(B, h, H, W):
    """ssba_forward_dense (Table 2's 0 % sparsity baseline) against the oracle's dense attention."""
    q, k, v, qd, kd, vd = _inputs(B, h, H, W, torch.bfloat16, seed=4)
    desc = api.SsbaDesc(B, h, H, W)
    O, lse = api.forward_dense(desc, qd, kd, vd)
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK
    O_o, lse_o = oracle.dense_forward(q, k, v)
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


def test_end_to_end_layer_with_gpu_mask():
    """build_mask then forward on the GPU (the path bench.py times), against the oracle
    forward run on the GPU's own lists."""
    H = W = 64
    q, k, v, qd, kd, vd = _inputs(1, 24, H, W, torch.bfloat16, seed=1)
    desc = api.SsbaDesc(1, 24, H, W, shift_r=4, shift_c=4, rho=0.8416)
    idx, cnt = api.build_mask(desc, qd, kd)
    O, lse = api.forward(desc, qd, kd, vd, idx, cnt)
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward(q, k, v, idx.cpu().numpy(), H, W, 8, (4, 4))
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


def test_status_word_reads_ok():
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK


# ----------------------------------------------------------------------------- split schedule
# With a forward workspace and lists of at least 24 blocks, the bf16 kernel gives each of
# its pipelines (two per SM) an equal share of key blocks and cuts the query blocks that
# straddle two shares, merging the two parts. 5 heads of a 64x64 grid are 320 query
# blocks: more than 2 x 152 pipelines and not a multiple of them, so shares end inside
# query blocks. rho = 0.5 keeps 32 of 64 blocks.
G = 64


def _split_inputs(seed, heads=5, rho=0.5, shift=(4, 4)):
    q, k, v, qd, kd, vd = _inputs(1, heads, G, G, torch.bfloat16, seed)
    desc = api.SsbaDesc(1, heads, G, G, shift_r=shift[0], shift_c=shift[1], rho=rho)
    idx_o, cnt_o = oracle.build_mask(q, k, G, G, 8, shift, rho)
    return desc, (q, k, v, qd, kd, vd), idx_o, cnt_o


def test_forward_split_and_whole_shares_agree_with_oracle():
    desc, (q, k, v, qd, kd, vd), idx_o, cnt_o = _split_inputs(0)
    assert idx_o.shape[-1] == 32
    O_o, lse_o = oracle.forward(q, k, v, idx_o, G, G, 8, (4, 4))
    idx_d, cnt_d = torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda()
    ws = torch.zeros(api.forward_workspace_bytes(desc), dtype=torch.uint8, device="cuda")
    for w in (ws, None):
        O, lse = api.forward(desc, qd, kd, vd, idx_d, cnt_d, workspace=w)
        torch.cuda.synchronize()
        check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


def test_forward_split_workspace_reused_across_calls():
    """Calls in a row on one workspace, each on new inputs: the boundary counters must
    be back at zero after every call, or a later call would merge stale parts."""
    ws = None
    for seed in (1, 2, 3):
        desc, (q, k, v, qd, kd, vd), idx_o, cnt_o = _split_inputs(seed, shift=(0, 0) if seed == 2 else (4, 4))
        if ws is None:
            ws = torch.zeros(api.forward_workspace_bytes(desc), dtype=torch.uint8, device="cuda")
        O, lse = api.forward(desc, qd, kd, vd, torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda(),
                             workspace=ws)
        torch.cuda.synchronize()
        O_o, lse_o = oracle.forward(q, k, v, idx_o, G, G, 8, (desc.shift_r, desc.shift_c))
        check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    counters = ws[: (2 * nsm + 1) * 16].view(torch.int32)
    assert int(counters.abs().sum()) == 0


def test_forward_split_ragged_counts():
    """Counts below the list length: many cut query blocks have an empty part (no block
    of the part's range is below the count), which must contribute nothing to the merge.
    The expected rows come from the oracle run on the lists truncated to each count."""
    desc, (q, k, v, qd, kd, vd), idx_o, _ = _split_inputs(4)
    keep = idx_o.shape[-1]
    Tb = G * G // 64
    choices = np.array([1, 9, 17, 25, keep], dtype=np.int32)
    items = np.arange(desc.B * desc.heads * Tb).reshape(desc.B, desc.heads, Tb)
    cnt = choices[(items * 7) % len(choices)]
    O, lse = api.forward(desc, qd, kd, vd, torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt).cuda())
    torch.cuda.synchronize()
    lab = oracle.partition(G, G, 8, (4, 4))
    O_ref = np.empty((desc.B, desc.heads, G * G, 64))
    lse_ref = np.empty((desc.B, desc.heads, G * G))
    for c in choices:
        O_c, lse_c = oracle.forward(q, k, v, np.ascontiguousarray(idx_o[..., :c]), G, G, 8, (4, 4))
        sel = cnt[:, :, lab] == c  # [B, heads, N]: rows whose query block has count c
        O_ref[sel] = O_c[sel]
        lse_ref[sel] = lse_c[sel]
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_ref, lse_ref, "bf16")


def test_forward_dense_split_schedule():
    q, k, v, qd, kd, vd = _inputs(1, 5, G, G, torch.bfloat16, seed=5)
    desc = api.SsbaDesc(1, 5, G, G)
    O_o, lse_o = oracle.dense_forward(q, k, v)
    for w in ("default", None):
        O, lse = api.forward_dense(desc, qd, kd, vd, workspace=w)
        torch.cuda.synchronize()
        check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


def test_forward_headline_whole_shares():
    """1024 px headline with and without a workspace (11-block lists: whole query blocks
    either way)."""
    q, k, v, qd, kd, vd = _inputs(1, 24, 64, 64, torch.bfloat16)
    desc = api.SsbaDesc(1, 24, 64, 64, shift_r=4, shift_c=4, rho=0.8416)
    idx_o, cnt_o = oracle.build_mask(q, k, 64, 64, 8, (4, 4), 0.8416)
    O, lse = api.forward(desc, qd, kd, vd, torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda(),
                         workspace=None)
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward(q, k, v, idx_o, 64, 64, 8, (4, 4))
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


# ----------------------------------------------------------------------------- text segment
# Algorithm 1 with its text segment: every image query also attends to all T_txt text keys
# (the token mask is padded with ones), and the image rows O[T_txt:] are returned.
def _joint_case(H, W, h, rho, shift, T_txt, seed=21, workspace="default"):
    q, k, v = synthetic.qkv(1, h, H * W, 64, torch.bfloat16, seed)
    kt, vt, _ = synthetic.qkv(1, h, T_txt, 64, torch.bfloat16, seed + 1)
    desc = api.SsbaDesc(1, h, H, W, shift_r=shift[0], shift_c=shift[1], rho=rho)
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, shift, rho)
    O, lse = api.forward_joint(desc, q.cuda(), k.cuda(), v.cuda(), kt.cuda(), vt.cuda(),
                               torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda(), workspace=workspace)
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward_joint(q, k, v, kt, vt, idx_o, H, W, 8, shift)
    return check_out(O.float().cpu().numpy(), lse.cpu().numpy(), O_o, lse_o, "bf16")


@pytest.mark.parametrize("T_txt,shift", [(77, (4, 4)), (256, (0, 0)), (5, (4, -4)), (0, (4, 4))])
def test_forward_joint_text(T_txt, shift):
    """Ragged (77 = 64 + 13), whole (256), shorter than one tile (5) and no text."""
    _joint_case(32, 32, 4, 0.75, shift, T_txt)


def test_forward_joint_headline_with_text():
    """1024 px headline geometry with a 256-token text prefix."""
    _joint_case(64, 64, 24, 0.8416, (4, 4), 256, seed=3)


@pytest.mark.parametrize("workspace", ["default", None])
def test_forward_joint_split_schedule(workspace):
    """A 1024-token text prefix makes 16 + 11 = 27 key blocks per query block, so with a
    workspace the pipelines take equal shares and cut query blocks; 320 query blocks."""
    _joint_case(64, 64, 5, 0.8416, (4, 4), 1024, seed=5, workspace=workspace)


# ----------------------------------------------------------------------------- backward
# Gradients of the sparse forward (fp32 outputs) against the fp64 oracle backward. The error
# is measured relative to the largest gradient of the tensor: with fp32 arithmetic and exact
# (fp32) O the bound is 1e-5 (measured about 1e-6); with bf16 inputs O is itself rounded to
# bf16 (2^-9 relative), which moves D = dO . O and through it every ds, so the bound is 5e-3
# (measured about 6e-4 at the 1024 px geometry).
BWD_TOL = {torch.float32: 1e-5, torch.bfloat16: 5e-3}


def _check_grads(got, ref, dtype):
    out = {}
    for name, g_, r in zip(("dQ", "dK", "dV"), got, ref):
        g_ = g_.cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(g_)), name
        rel = float(np.abs(g_ - r).max() / max(1.0, np.abs(r).max()))
        out[name] = rel
        assert rel <= BWD_TOL[dtype], (name, rel)
    return out


def _bwd_case_gpu(B, h, H, W, rho, shift, dtype, seed):
    q, k, v = synthetic.qkv(B, h, H * W, 64, dtype, seed)
    go = synthetic.qkv(B, h, H * W, 64, dtype, seed + 100)[0]
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, shift, rho)
    O_o, lse_o = oracle.forward(q, k, v, idx_o, H, W, 8, shift)
    desc = api.SsbaDesc(B, h, H, W, shift_r=shift[0], shift_c=shift[1], rho=rho, dtype=dtype)
    grads = api.backward(desc, q.cuda(), k.cuda(), v.cuda(), torch.from_numpy(O_o).to(dtype).cuda(),
                         torch.from_numpy(lse_o).float().cuda(), go.cuda(), torch.from_numpy(idx_o).cuda(),
                         torch.from_numpy(cnt_o).cuda())
    torch.cuda.synchronize()
    ref = oracle.backward(q, k, v, go, idx_o, H, W, 8, shift)
    return _check_grads(grads, ref, dtype)


@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (3, -5)])
@pytest.mark.parametrize("rho", [0.75, 0.0])
def test_backward_fp32_tiny(shift, rho):
    _bwd_case_gpu(1, 2, 16, 16, rho, shift, torch.float32, 30)


@pytest.mark.parametrize("H,W,h,rho,shift", [(32, 32, 4, 0.75, (4, 4)), (64, 64, 4, 0.8416, (4, 4)),
                                            (24, 40, 3, 0.6, (4, -4)),
                                            # one, two and three kept blocks a row: the pipelined
                                            # loops with fewer pairs than tile buffers
                                            (16, 16, 4, 0.75, (4, 4)), (16, 16, 4, 0.5, (3, -5)),
                                            (16, 24, 2, 0.5, (0, 0))])
def test_backward_bf16(H, W, h, rho, shift):
    _bwd_case_gpu(1, h, H, W, rho, shift, torch.bfloat16, 31)


@pytest.mark.parametrize("B,H,W,h,rho,shift", [(2, 32, 32, 3, 0.75, (4, 4)),
                                              # 256 blocks a head (the 2048 px grid): long rows
                                              # and key blocks kept by many query blocks
                                              (1, 128, 128, 2, 0.84, (4, 4))])
def test_backward_bf16_batches_and_long_rows(B, H, W, h, rho, shift):
    _bwd_case_gpu(B, h, H, W, rho, shift, torch.bfloat16, 34)


def test_backward_is_deterministic():
    """Repeated calls give bitwise-equal gradients: no atomics, and the work counter only decides
    which CTA runs an item, not the order of any sum (1024 px layer, 24 heads, shift 4)."""
    H = W = 64
    q, k, v = synthetic.qkv(1, 24, H * W, 64, torch.bfloat16, 33)
    go = synthetic.qkv(1, 24, H * W, 64, torch.bfloat16, 133)[0].cuda()
    desc = api.SsbaDesc(1, 24, H, W, shift_r=4, shift_c=4, rho=0.8416)
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    idx, cnt = api.build_mask(desc, qd, kd)
    O, lse = api.forward(desc, qd, kd, vd, idx, cnt)
    first = [g.clone() for g in api.backward(desc, qd, kd, vd, O, lse, go, idx, cnt)]
    for _ in range(3):
        again = api.backward(desc, qd, kd, vd, O, lse, go, idx, cnt)
        torch.cuda.synchronize()
        for a, b in zip(first, again):
            assert torch.equal(a, b)
    assert api.get_status() == api.SSBA_OK


def test_backward_after_gpu_forward():
    """The training order: GPU mask, GPU forward, then the backward on the forward's own O
    and lse, against the oracle backward on the same lists."""
    H = W = 32
    q, k, v = synthetic.qkv(1, 4, H * W, 64, torch.bfloat16, 32)
    go = synthetic.qkv(1, 4, H * W, 64, torch.bfloat16, 132)[0]
    desc = api.SsbaDesc(1, 4, H, W, shift_r=4, shift_c=4, rho=0.75)
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    idx, cnt = api.build_mask(desc, qd, kd)
    O, lse = api.forward(desc, qd, kd, vd, idx, cnt)
    grads = api.backward(desc, qd, kd, vd, O, lse, go.cuda(), idx, cnt)
    torch.cuda.synchronize()
    ref = oracle.backward(q, k, v, go, idx.cpu().numpy(), H, W, 8, (4, 4))
    _check_grads(grads, ref, torch.bfloat16)
