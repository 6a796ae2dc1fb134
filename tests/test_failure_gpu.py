"""Failure detection on the GPU, without a fault: every barrier wait of the tensor-core
forward is bounded in wall time. A test hook announces one K tile copy that it never
issues, so the waits on that tile run out; the kernel must stop, drain what it issued,
free its tensor memory and report SSBA_ERR_TIMEOUT in the device status word, and the
CUDA context must stay usable (a normal forward right after matches the oracle)."""
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
