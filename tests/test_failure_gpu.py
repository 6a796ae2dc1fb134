"""Failure detection on the GPU, without a fault: every barrier wait of the tensor-core
forward is bounded in wall time. A test hook announces one K tile copy that it never
issues, so the waits on that tile run out; the kernel must stop, drain what it issued,
free its tensor memory and report SSBA_ERR_TIMEOUT in the device status word, and the
CUDA context must stay usable (a normal forward right after matches the oracle). A second
hook makes one CTA of the fused launch withhold its arrival at the grid barrier, so that
every CTA's barrier wait runs out, with the same requirements. A third makes one CTA of the
persistent backward announce a pair's tile copies without issuing them."""
import pytest
import torch

import oracle
from paper_2605_15684_gb300 import api, build, synthetic
from tests.parity import check_out

pytestmark = pytest.mark.gpu


def test_timed_out_wait_reports_status_and_context_survives():
    build.build()
    api.load_library()
    H = W = 32
    q, k, v = synthetic.qkv(1, 4, H * W, 64, torch.bfloat16, 11)
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    desc = api.SsbaDesc(1, 4, H, W, shift_r=4, shift_c=4, rho=0.75)
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, (4, 4), 0.75)
    idx, cnt = torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda()
    O = torch.empty_like(qd)
    lse = torch.empty(1, 4, H * W, device="cuda")
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK  # read-and-clear: start clean

    api.test_forward_timeout(desc, qd, kd, vd, idx, cnt, O, lse, budget_ns=2_000_000)
    torch.cuda.synchronize()  # the kernel returns: no hang, no CUDA error
    assert api.get_status() == api.SSBA_ERR_TIMEOUT
    assert api.get_status() == api.SSBA_OK  # cleared by the read

    O2, lse2 = api.forward(desc, qd, kd, vd, idx, cnt)
    torch.cuda.synchronize()
    O_o, lse_o = oracle.forward(q, k, v, idx_o, H, W, 8, (4, 4))
    check_out(O2.float().cpu().numpy(), lse2.cpu().numpy(), O_o, lse_o, "bf16")
    assert api.get_status() == api.SSBA_OK


def test_grid_barrier_timeout_reports_status_and_context_survives():
    build.build()
    api.load_library()
    H = W = 64
    q, k, v = synthetic.qkv(1, 24, H * W, 64, torch.bfloat16, 12)
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    desc = api.SsbaDesc(1, 24, H, W, shift_r=4, shift_c=4, rho=0.8416)
    keep = api.keep_count(desc)
    Tb = H * W // 64
    qb = torch.empty(1, 24, Tb, 64, device="cuda")
    kb = torch.empty_like(qb)
    idx = torch.empty(1, 24, Tb, keep, dtype=torch.int32, device="cuda")
    cnt = torch.empty(1, 24, Tb, dtype=torch.int32, device="cuda")
    O = torch.empty_like(qd)
    lse = torch.empty(1, 24, H * W, device="cuda")
    ws = torch.zeros(api.forward_workspace_bytes(desc), dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK  # read-and-clear: start clean

    api.test_fused_timeout(desc, qd, kd, vd, qb, kb, idx, cnt, O, lse, ws, budget_ns=2_000_000)
    torch.cuda.synchronize()  # every CTA gives up at the barrier and returns: no hang, no CUDA error
    assert api.get_status() == api.SSBA_ERR_TIMEOUT
    assert api.get_status() == api.SSBA_OK

    # the CTAs that arrived left their count in the barrier words (none departed), so the
    # workspace must be zeroed again before the next call, as the header says
    assert int(ws[-256:].count_nonzero()) > 0
    ws.zero_()
    O2, l2, i2, c2, qb2, kb2 = api.forward_fused(desc, qd, kd, vd, workspace=ws)
    qb3, kb3 = api.pool_blocks(desc, qd, kd)
    O3, l3, i3, c3 = api.forward_select(desc, qd, kd, vd, qb3, kb3)
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK
    assert torch.equal(i2, i3) and torch.equal(O2, O3) and torch.equal(l2, l3)
    assert int(ws[-256:].count_nonzero()) == 0


def test_backward_timeout_reports_status_and_context_survives():
    """CTA 0 of the persistent backward never receives its first pair's tiles: its issuers'
    waits run out, it drains and reports SSBA_ERR_TIMEOUT, the other CTAs finish; a normal
    backward right after matches the oracle."""
    build.build()
    api.load_library()
    H = W = 32
    q, k, v = synthetic.qkv(1, 4, H * W, 64, torch.bfloat16, 13)
    go = synthetic.qkv(1, 4, H * W, 64, torch.bfloat16, 113)[0]
    desc = api.SsbaDesc(1, 4, H, W, shift_r=4, shift_c=4, rho=0.75)
    qd, kd, vd, god = q.cuda(), k.cuda(), v.cuda(), go.cuda()
    idx_o, cnt_o = oracle.build_mask(q, k, H, W, 8, (4, 4), 0.75)
    O_o, lse_o = oracle.forward(q, k, v, idx_o, H, W, 8, (4, 4))
    idx, cnt = torch.from_numpy(idx_o).cuda(), torch.from_numpy(cnt_o).cuda()
    O = torch.from_numpy(O_o).to(torch.bfloat16).cuda()
    lse = torch.from_numpy(lse_o).float().cuda()
    torch.cuda.synchronize()
    assert api.get_status() == api.SSBA_OK

    api.test_backward_timeout(desc, qd, kd, vd, O, lse, god, idx, cnt, budget_ns=2_000_000)
    torch.cuda.synchronize()  # the kernel returns: no hang, no CUDA error
    assert api.get_status() == api.SSBA_ERR_TIMEOUT
    assert api.get_status() == api.SSBA_OK

    grads = api.backward(desc, qd, kd, vd, O, lse, god, idx, cnt)
    torch.cuda.synchronize()
    ref = oracle.backward(q, k, v, go, idx_o, H, W, 8, (4, 4))
    for got, want in zip(grads, ref):  # the bf16 bound of the parity tests
        g = got.cpu().double().numpy()
        assert abs(g - want).max() / max(1.0, abs(want).max()) <= 5e-3
    assert api.get_status() == api.SSBA_OK
