"""GPU parity of the fused QKV projection + RoPE + block pooling (ssba_qkv_rope_pool) and of
the selection from block means (ssba_select_mask), through the C-ABI, against the oracle.

Tolerances (derived, not fitted):
  * Q, K, V: the GPU accumulates the Dm products in fp32 on the tensor cores; the bound
    allows 2^-12 * sum_k |x_k w_k| for that (well above Dm * 2^-24 for Dm <= 1536), doubled
    for a RoPE pair (a rotation mixes the errors of two channels), plus the bf16 rounding
    of the result, 2^-8 * |ref|;
  * q_b, k_b: means of the GPU's own bf16 Q and K, 64 fp32 additions: 2^-18 * mean|q|;
  * lists: bit-exact on the GPU's own scores, margin-gated against the oracle (tests/parity.py).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_15684_gb300 import api, build, synthetic
from tests.parity import check_mask

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    api.load_library()
    yield
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK


def _run(B, heads, H, W, shift, rho=0.75, seed=0, bias=True):
    Dm = heads * 64
    X, Wq, b = synthetic.projection_inputs(B, H * W, Dm, seed)
    desc = api.SsbaDesc(B, heads, H, W, shift_r=shift[0], shift_c=shift[1], rho=rho, dtype=torch.bfloat16)
    Q, K, V, qb, kb = api.qkv_rope_pool(desc, X.cuda(), Wq.cuda(), b.cuda() if bias else None)
    torch.cuda.synchronize()
    return desc, (X, Wq, b if bias else None), (Q.cpu(), K.cpu(), V.cpu(), qb.cpu(), kb.cpu())


def _bound(X, Wq, heads, H, W):
    """Per output element: 2^-12 * sum_k |x_k w_k|, as [3, B, heads, N, 64], RoPE pairs doubled."""
    M = np.abs(X.double().numpy()) @ np.abs(Wq.double().numpy()).T  # [B, N, 3 Dm]
    B, N, _ = M.shape
    M = M.reshape(B, N, 3, heads, 64).transpose(2, 0, 3, 1, 4) * 2.0 ** -12
    pair = np.maximum(M[..., 0::2], M[..., 1::2])
    M[:2, ..., 0::2] = 2 * pair[:2]
    M[:2, ..., 1::2] = 2 * pair[:2]
    return M


def _check_qkv(got, ref, acc_bound):
    got = got.double().numpy()
    tol = 2.0 ** -8 * np.abs(ref) + acc_bound + 1e-6
    err = np.abs(got - ref)
    assert np.all(err <= tol), f"max excess {float(np.max(err - tol)):.3e}"


def _check_pooled(qb, Q, H, W, shift):
    ref = oracle.pooled_blocks(Q.double().numpy(), H, W, 8, shift)
    mag = oracle.pooled_blocks(np.abs(Q.double().numpy()), H, W, 8, shift)
    err = np.abs(qb.double().numpy() - ref)
    assert np.all(err <= 2.0 ** -18 * mag + 1e-12), f"max {float(err.max()):.3e}"


@pytest.mark.parametrize("B,heads,H,W,shift", [
    (1, 4, 16, 16, (0, 0)),     # one N tile per Q/K/V, two M tiles
    (1, 4, 16, 16, (4, 4)),     # shifted: every window crosses an edge
    (2, 3, 24, 16, (4, -4)),    # 3 Dm = 576: a partial N tile, heads straddle tiles
    (1, 2, 8, 24, (0, 4)),      # Tb = 3: the last M tile holds one window
    (1, 5, 40, 24, (-4, 0)),    # 15 windows, five heads
])
def test_qkv_rope_pool_matches_oracle(B, heads, H, W, shift):
    desc, (X, Wq, b), (Q, K, V, qb, kb) = _run(B, heads, H, W, shift, seed=B * 100 + heads)
    Qo, Ko, Vo = oracle.qkv_rope(X.double().numpy(), Wq.double().numpy(), b.double().numpy(), heads, H, W)
    acc = _bound(X, Wq, heads, H, W)
    _check_qkv(Q, Qo, acc[0])
    _check_qkv(K, Ko, acc[1])
    _check_qkv(V, Vo, acc[2])
    _check_pooled(qb, Q, H, W, shift)
    _check_pooled(kb, K, H, W, shift)


def test_qkv_without_bias_or_pooling():
    desc, (X, Wq, _), (Q, K, V, qb, kb) = _run(1, 2, 16, 16, (4, 4), seed=7, bias=False)
    Qo, Ko, Vo = oracle.qkv_rope(X.double().numpy(), Wq.double().numpy(), None, 2, 16, 16)
    acc = _bound(X, Wq, 2, 16, 16)
    _check_qkv(Q, Qo, acc[0])
    _check_qkv(V, Vo, acc[2])
    Q2, K2, V2, n1, n2 = api.qkv_rope_pool(desc, X.cuda(), Wq.cuda(), None, pooled=False)
    torch.cuda.synchronize()
    assert n1 is None and n2 is None
    assert torch.equal(Q2.cpu(), Q) and torch.equal(K2.cpu(), K) and torch.equal(V2.cpu(), V)


def test_qkv_1024px_sampled_and_pooling_everywhere():
    """The 1024 px projection (4096 tokens, 24 heads, Dm = 1536): every pooled mean, and the
    outputs of 512 sampled tokens, against the oracle's projection of those tokens."""
    heads, H, W, shift = 24, 64, 64, (4, 4)
    desc, (X, Wq, b), (Q, K, V, qb, kb) = _run(1, heads, H, W, shift, seed=11)
    _check_pooled(qb, Q, H, W, shift)
    _check_pooled(kb, K, H, W, shift)
    rng = np.random.default_rng(12)
    toks = np.sort(rng.choice(H * W, 512, replace=False))
    # the oracle on the sampled rows: project the rows, turn them at their own positions
    Xs = X.double().numpy()[:, toks]
    Y = Xs @ Wq.double().numpy().T + b.double().numpy()
    Y = Y.reshape(1, len(toks), 3, heads, 64).transpose(2, 0, 3, 1, 4)
    full = np.zeros((3, 1, heads, H * W, 64))
    full[:, :, :, toks] = Y
    Qo = oracle.rope_2d(full[0], H, W)[:, :, toks]
    Ko = oracle.rope_2d(full[1], H, W)[:, :, toks]
    Vo = full[2][:, :, toks]
    M = np.abs(Xs) @ np.abs(Wq.double().numpy()).T
    M = M.reshape(1, len(toks), 3, heads, 64).transpose(2, 0, 3, 1, 4) * 2.0 ** -12
    pair = np.maximum(M[..., 0::2], M[..., 1::2])
    M[:2, ..., 0::2] = 2 * pair[:2]
    M[:2, ..., 1::2] = 2 * pair[:2]
    _check_qkv(Q[:, :, toks], Qo, M[0])
    _check_qkv(K[:, :, toks], Ko, M[1])
    _check_qkv(V[:, :, toks], Vo, M[2])


@pytest.mark.parametrize("H,W,shift,rho", [(16, 16, (4, 4), 0.75), (64, 64, (4, 4), 0.8416), (40, 24, (0, 0), 0.6)])
def test_select_mask_from_pooled(H, W, shift, rho):
    """Selection from the fused path's means: exact on the GPU's own scores, and against the
    oracle's mask of the GPU's Q and K (tie policy of tests/parity.py)."""
    heads = 4
    desc, _, (Q, K, V, qb, kb) = _run(1, heads, H, W, shift, rho=rho, seed=21)
    idx, cnt, S = api.select_mask(desc, qb.cuda(), kb.cuda(), scores=True)
    torch.cuda.synchronize()
    idx_o, cnt_o, S_o = oracle.build_mask(Q.double().numpy(), K.double().numpy(), H, W, 8, shift, rho,
                                          return_scores=True)
    keep = oracle.keep_count(H * W // 64, rho)
    near = check_mask(idx.cpu().numpy(), cnt.cpu().numpy(), S.cpu().numpy(), S_o, idx_o, keep)
    assert near < 0.1 * heads * (H * W // 64)


def test_fused_path_feeds_the_forward():
    """Projection -> selection -> sparse attention, all on the GPU, against the oracle's
    forward on the GPU's own Q, K, V and lists (bf16 tolerance)."""
    from tests.parity import check_out
    heads, H, W, shift = 4, 32, 32, (4, 4)
    desc, _, (Q, K, V, qb, kb) = _run(1, heads, H, W, shift, rho=0.8416, seed=31)
    idx, cnt = api.select_mask(desc, qb.cuda(), kb.cuda())
    O, lse = api.forward(desc, Q.cuda(), K.cuda(), V.cuda(), idx, cnt)
    torch.cuda.synchronize()
    Oo, lo = oracle.forward(Q.double().numpy(), K.double().numpy(), V.double().numpy(), idx.cpu().numpy(), H, W, 8,
                            shift)
    check_out(O.float().cpu().numpy(), lse.cpu().numpy(), Oo, lo, "bf16")
