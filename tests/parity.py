"""Comparison helpers shared by the GPU parity tests (test infrastructure).

Tolerances (written here, used by every parity test):
  * block indices and counts: bit-exact (see check_mask for the tie policy);
  * O from fp32 inputs: max-abs <= 1e-4; lse max-abs <= 1e-4;
  * O from bf16 inputs: max-abs <= 2e-2 and mean-abs <= 5e-3; lse max-abs <= 1e-2.
"""
from __future__ import annotations

import numpy as np

import oracle

TOL = {
    "fp32": dict(o_max=1e-4, o_mean=1e-4, lse_max=1e-4),
    "bf16": dict(o_max=2e-2, o_mean=5e-3, lse_max=1e-2),
}


def check_mask(idx_gpu, cnt_gpu, S_gpu, S_oracle, idx_oracle, keep, rel_margin=1e-4):
    """Tie policy for the kept-block lists.

    1. Selection stage, exact: the oracle's gate run on the GPU's own fp32 S (widened
       exactly to fp64) must reproduce the GPU lists bit for bit, in every row.
    2. End to end, margin-gated: where the oracle's fp64 gap between the keep-th and
       (keep+1)-th largest S of a row exceeds rel_margin * max|S_row|, the GPU list
       must equal the oracle's bit for bit; rows inside the margin must still be a
       valid top-keep set of the oracle's S within that margin.
    Returns the number of rows that fell inside the margin.
    """
    idx_gpu = np.asarray(idx_gpu)
    cnt_gpu = np.asarray(cnt_gpu)
    S_gpu = np.asarray(S_gpu, dtype=np.float64)
    Tb = S_oracle.shape[-1]
    k_drop = Tb - keep
    assert np.all(cnt_gpu == keep)
    flat_gpu = idx_gpu.reshape(-1, Tb, keep)
    flat_Sg = S_gpu.reshape(-1, Tb, Tb)
    flat_So = np.asarray(S_oracle, dtype=np.float64).reshape(-1, Tb, Tb)
    flat_io = np.asarray(idx_oracle).reshape(-1, Tb, keep)
    near = 0
    for s in range(flat_gpu.shape[0]):
        # 1. exact selection on the GPU's scores
        assert np.array_equal(oracle.gate(flat_Sg[s], k_drop), flat_gpu[s]), f"selection differs in slice {s}"
        for i in range(Tb):
            row = flat_So[s, i]
            srt = np.sort(row)[::-1]
            gap = srt[keep - 1] - srt[keep] if keep < Tb else np.inf
            tau = rel_margin * np.max(np.abs(row))
            if gap > tau:
                assert np.array_equal(flat_gpu[s, i], flat_io[s, i]), f"slice {s} row {i}"
            else:
                near += 1
                kept = flat_gpu[s, i]
                dropped = np.setdiff1d(np.arange(Tb), kept)
                assert len(np.unique(kept)) == keep
                if len(dropped):
                    assert row[kept].min() >= row[dropped].max() - tau
    return near


def check_out(O_gpu, lse_gpu, O_ref, lse_ref, kind: str):
    tol = TOL[kind]
    O_gpu = np.asarray(O_gpu, dtype=np.float64)
    lse_gpu = np.asarray(lse_gpu, dtype=np.float64)
    assert np.all(np.isfinite(O_gpu)) and np.all(np.isfinite(lse_gpu))
    err = np.abs(O_gpu - O_ref)
    lerr = np.abs(lse_gpu - lse_ref)
    stats = dict(o_max=float(err.max()), o_mean=float(err.mean()), lse_max=float(lerr.max()))
    assert stats["o_max"] <= tol["o_max"], stats
    assert stats["o_mean"] <= tol["o_mean"], stats
    assert stats["lse_max"] <= tol["lse_max"], stats
    return stats
