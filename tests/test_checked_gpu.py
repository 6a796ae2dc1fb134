"""The checked build of the library (build.py variant "checked", -DSSBA_CHECKED): the attention
kernel tests the invariants of the index lists it reads (labels in [0, Tb), rows strictly
ascending, counts in [0, keep]) and reports a violation as SSBA_ERR_CHECK in the device status
word. Bad values are still clamped into range, as in the default build, so these inputs are
safe to run. The binding loads one library per process, so the checks run in a child process."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys
sys.path.insert(0, sys.argv[1])
import torch
from paper_2605_15684_gb300 import api, build, synthetic
api.load_library(build.build(variant="checked"))
H = W = 32
desc = api.SsbaDesc(1, 4, H, W, shift_r=4, shift_c=4, rho=0.75)
q, k, v = (t.cuda() for t in synthetic.qkv(1, 4, H * W, 64, torch.bfloat16, 3))
idx, cnt = api.build_mask(desc, q, k)
O, lse = api.forward(desc, q, k, v, idx, cnt)
torch.cuda.synchronize()
assert api.get_status() == api.SSBA_OK, "valid lists flagged"
keep = idx.shape[-1]
cases = []
bad = idx.clone(); bad[0, 1, 3, keep - 1] = desc.Tb + 5; cases.append(("label past Tb", bad, cnt))
bad = idx.clone(); bad[0, 2, 0, :2] = bad[0, 2, 0, :2].flip(0); cases.append(("descending row", bad, cnt))
badc = cnt.clone(); badc[0, 0, 7] = keep + 1; cases.append(("count above keep", idx, badc))
for name, i2, c2 in cases:
    api.forward(desc, q, k, v, i2, c2, workspace=None)
    torch.cuda.synchronize()
    st = api.get_status()
    assert st == api.SSBA_ERR_CHECK, (name, st)
# the fused timed path on valid inputs stays clean
api.forward_fused(desc, q, k, v)
torch.cuda.synchronize()
assert api.get_status() == api.SSBA_OK
print("checked build ok")
"""


@pytest.mark.gpu
def test_checked_build_reports_broken_lists():
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "checked build ok" in r.stdout
