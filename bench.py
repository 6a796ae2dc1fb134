#!/usr/bin/env python3
"""Benchmark of the SSBA forward (mask build + block-sparse attention) on GB300.

A step is one pass of the whole hot path over one batch: the 24 SSBA layers of the
1024 px DiT (64 x 64 image tokens, B=1, 24 heads x 64, rho = 0.8416 -> keep 11 of 64
blocks per query block), layer l with window shift (0,0) if l is even else (4,4); each
layer is one launch (ssba_forward_fused) that pools the block means from its own Q/K,
computes the affinities, selects the kept blocks and runs the block-sparse forward. The
pooling as a launch of its own (ssba_pool_blocks + ssba_forward_select) and the two-launch
path (ssba_build_mask + ssba_forward) are measured beside it, outside the timed region. Each
layer has its own seeded synthetic Q/K/V (906 MB in all), so every layer's inputs are
cold in L2 when it runs.

Prints one JSON line. value = effective TFLOP/s counting only the kept blocks
(4 * B * heads * Tb * keep * 64 * 64 * head_dim per layer) over the whole step. Beside it:
`roofline` (the fused launch against the bf16 peak), `roofline_mask` (the mask kernel of
ssba_build_mask against the HBM peak), `roofline_pool`, `configs_sweep` (the paper's other
workloads, each on the fused launch and, as `two_call_ms_per_layer`, through
ssba_build_mask + ssba_forward), the same-build dense kernel, the backward, the NEXT rows'
kernels, `e2e`, `cpu_baseline` and the clocks sampled during the timed region.
``--impl reference`` times the CPU oracle on the host cores instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "SSBA fwd latency (ms) and effective TFLOP/s @4096 tok, 84% sparse, bf16"
ATTN_SOURCES = ("paper_2605_15684_gb300/csrc/attn_tc.cu", "paper_2605_15684_gb300/csrc/ptx.cuh",
                "paper_2605_15684_gb300/csrc/window.cuh")
ATTN_PROFILE = os.path.join(ROOT, "profiles", "ssba_attn_tc_kernel_1024px.md")
MASK_SOURCES = ("paper_2605_15684_gb300/csrc/mask.cu", "paper_2605_15684_gb300/csrc/select.cuh",
                "paper_2605_15684_gb300/csrc/ptx.cuh")
MASK_PROFILE = os.path.join(ROOT, "profiles", "ssba_mask_fused_kernel_1024px.md")


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--layers", type=int, default=24)
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    return ap.parse_args()


# ----------------------------------------------------------------------------- workload
def workload():
    from paper_2605_15684_gb300 import synthetic
    return synthetic.PX1024


def layer_shift(l: int):
    return (0, 0) if l % 2 == 0 else (4, 4)


def max_over_ranks(x: float, world: int, device=None) -> float:
    """The largest x over all ranks (the slowest rank's time); x itself on one rank."""
    if world <= 1:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_tflops(world: int, flops_per_rank: float, seconds: float) -> float:
    """Whole-job rate: every rank does flops_per_rank of independent work; the job takes
    as long as its slowest rank (seconds)."""
    return world * flops_per_rank / seconds / 1e12


def mask_launches(head_dim: int, Tb: int, blk: int = 8) -> int:
    """Kernels one ssba_build_mask call launches: the fused build (head_dim 64, 8x8 blocks,
    at most 256 blocks) is one, the pooling + selection pair is two."""
    return 1 if (head_dim == 64 and blk == 8 and Tb <= 256) else 2


def kept_flops(B, h, Tb, keep, d, blk=8):
    """QK^T plus PV over the kept blocks only (2 * 2 * rows * keys * d)."""
    return 4.0 * B * h * Tb * keep * (blk * blk) * (blk * blk) * d


def config_dict(w, keep, layers):
    Tb = w.N // 64
    return {
        "workload": f"{w.name} x{layers} layers, shifts (0,0)/(4,4) alternating, mask rebuilt per layer "
                    f"(pooling, selection and attention in one launch per layer)",
        "B": w.B, "heads": w.heads, "grid": [w.H_tok, w.W_tok], "N": w.N, "head_dim": w.head_dim,
        "block": 8, "rho": w.rho, "Tb": Tb, "keep": keep,
        "realized_sparsity": round((Tb - keep) / Tb, 6), "layers": layers,
        "l2": "inputs larger than L2: each layer has its own Q/K/V, "
              f"{layers * 3 * w.B * w.heads * w.N * w.head_dim * 2 / 1e6:.0f} MB per step",
    }


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampled every 50 ms in a background process; samples are stamped with
    the host clock on arrival so the timed window can be selected afterwards."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.samples = []
        self.proc = None
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50"]
        if gpu_id:
            cmd += ["-i", gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.strip().split(",")]
            if len(parts) < 8:
                continue
            try:
                self.samples.append((time.time(), float(parts[0]), float(parts[1]), parts[2], parts[3:]))
            except ValueError:
                continue

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        win = [s for s in self.samples if t0 <= s[0] <= t1] or self.samples
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = set()
        for s in win:
            for nm, flag in zip(names, s[4][1:]):
                if flag.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(s[1] for s in win), "sm_max_mhz": max(s[2] for s in win),
                "reasons": sorted(reasons), "samples": len(win),
                "power_w_max": max((float(s[3]) for s in win if s[3].replace(".", "", 1).isdigit()),
                                   default=None)}


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the platform string)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().startswith("Model name:"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith("model name"):
                    return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.machine() + " " + platform.processor()


# ----------------------------------------------------------------------------- roofline helpers
def measured_peaks_sustained() -> float:
    """The measured sustained dense bf16 rate (for a kernel timed inside a long step)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops_sustained"])
    except Exception:
        return 1700.0


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return j.get("hbm_gbs", 6800.0), j.get("bf16_tflops", 1900.0), "measured"
    return 6800.0, 1900.0, "fallback"


def profiled_traffic(profile=ATTN_PROFILE, sources=ATTN_SOURCES):
    """DRAM bytes per launch of a kernel from its committed ncu summary, if the kernel's
    sources are unchanged since the capture (else None)."""
    if not os.path.exists(profile):
        return None
    text = open(profile).read()
    m_b = re.search(r"dram_bytes_per_launch:\s*([0-9]+)", text)
    m_h = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    if not m_b or not m_h:
        return None
    h = hashlib.sha256()
    for rel in sources:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return int(m_b.group(1)) if h.hexdigest() == m_h.group(1) else None


# ----------------------------------------------------------------------------- reference arm
def oracle_sample(w, heads_sample: int, seed: int = 0):
    """Times the fp64 CPU oracle (mask + forward) on `heads_sample` heads of one layer."""
    import oracle
    from paper_2605_15684_gb300 import synthetic
    q, k, v = synthetic.qkv(1, heads_sample, w.N, w.head_dim, w.dtype, seed, w.std)
    Qd, Kd, Vd = (oracle._f64(x) for x in (q, k, v))
    shift = layer_shift(0)
    t0 = time.perf_counter()
    idx, _ = oracle.build_mask(Qd, Kd, w.H_tok, w.W_tok, 8, shift, w.rho)
    oracle.forward(Qd, Kd, Vd, idx, w.H_tok, w.W_tok, 8, shift)
    dt = time.perf_counter() - t0
    Tb = w.N // 64
    keep = idx.shape[-1]
    return kept_flops(1, heads_sample, Tb, keep, w.head_dim) / dt / 1e12, dt


def run_reference(args, rank):
    if rank != 0:
        return
    import oracle
    w = workload()
    threads = oracle.max_threads()
    heads_sample = max(1, min(w.heads, threads))
    Tb = w.N // 64
    keep = oracle.keep_count(Tb, w.rho)
    for _ in range(args.warmup):
        oracle_sample(w, heads_sample)
    rates, times = [], []
    for s in range(args.steps):
        r, dt = oracle_sample(w, heads_sample, seed=s)
        rates.append(r)
        times.append(dt)
    total_flops = kept_flops(1, heads_sample, Tb, keep, w.head_dim) * args.steps
    value = total_flops / sum(times) / 1e12
    sample = (f"{heads_sample} of {w.heads} heads of layer 0 per step (mask + forward), "
              f"OpenMP over heads")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * sum(times) / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_dict(w, keep, args.layers),
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": min(threads, heads_sample),
                         "nproc": os.cpu_count(), "cpu_model": cpu_model(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- our arm
def run_ours(args, rank, world):
    import torch
    from paper_2605_15684_gb300 import api, build, synthetic

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    if rank == 0 or world == 1:
        build.build()
    if world > 1:
        torch.distributed.barrier()
    api.load_library()
    w = workload()
    L = args.layers
    Tb = w.N // 64
    descs = [api.SsbaDesc(w.B, w.heads, w.H_tok, w.W_tok, w.head_dim, 8, *layer_shift(l), w.rho, w.dtype)
             for l in range(L)]
    keep = api.keep_count(descs[0])
    shp = (w.B, w.heads, w.N, w.head_dim)

    # per-layer inputs: seed = layer + 1000 * rank (independent problems per rank)
    host_qkv = [synthetic.qkv(w.B, w.heads, w.N, w.head_dim, w.dtype, seed=l + 1000 * rank, std=w.std)
                for l in range(L)]
    Qs = [h[0].to(dev) for h in host_qkv]
    Ks = [h[1].to(dev) for h in host_qkv]
    Vs = [h[2].to(dev) for h in host_qkv]
    idx = [torch.empty((w.B, w.heads, Tb, keep), dtype=torch.int32, device=dev) for _ in range(L)]
    cnt = [torch.empty((w.B, w.heads, Tb), dtype=torch.int32, device=dev) for _ in range(L)]
    Os = [torch.empty(shp, dtype=w.dtype, device=dev) for _ in range(L)]
    lses = [torch.empty(shp[:3], dtype=torch.float32, device=dev) for _ in range(L)]
    ws = torch.empty(api.mask_workspace_bytes(descs[0]), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    pshp = (w.B, w.heads, Tb, w.head_dim)
    qbs = [torch.empty(pshp, dtype=torch.float32, device=dev) for _ in range(L)]
    kbs = [torch.empty(pshp, dtype=torch.float32, device=dev) for _ in range(L)]
    # the timed path: pooling, selection and attention in one launch per layer (ssba_forward_fused)
    layers = [api.BoundSelectLayer(descs[l], Qs[l], Ks[l], Vs[l], qbs[l], kbs[l], idx[l], cnt[l], Os[l], lses[l],
                                   stream) for l in range(L)]
    # the two-launch path (mask kernel, then the forward on its lists), measured beside it
    layers2 = [api.BoundLayer(descs[l], Qs[l], Ks[l], Vs[l], idx[l], cnt[l], Os[l], lses[l], ws, stream)
               for l in range(L)]

    def step(ev=None):
        for l, ly in enumerate(layers):
            if ev is not None:
                ev[0][l].record(stream)
            ly.fused()
            if ev is not None:
                ev[1][l].record(stream)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    st = torch.zeros(1, dtype=torch.int32)
    st[0] = api.get_status()
    if int(st[0]) != api.SSBA_OK:
        raise RuntimeError(f"device status {int(st[0])} after warm-up")

    # ---- timed region: K steps, per-kernel events on the launching stream
    K = args.steps
    evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(L)] for _ in range(2)] for _ in range(K)]
    gpu_id = None
    try:
        gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
        gpu_id = gpu_id if gpu_id.startswith("GPU-") else "GPU-" + gpu_id
    except Exception:
        gpu_id = None
    clocks = ClockSampler(gpu_id)
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    # events only around the K steps: an event recorded between two launches ends the overlap
    # that programmatic dependent launch gives them (measured: about 5 % of the step)
    wall0 = time.time()
    t_start.record(stream)
    for s in range(K):
        step()
    t_end.record(stream)
    torch.cuda.synchronize()
    wall1 = time.time()
    if world > 1:
        torch.distributed.barrier()
    time.sleep(0.1)
    clocks.stop()
    ms_total = t_start.elapsed_time(t_end)
    ms_total = max_over_ranks(ms_total, world, dev)
    ms_step = ms_total / K
    # ---- the same K steps again with an event around every launch: the kernels' durations
    for s in range(K):
        step(evs[s])
    torch.cuda.synchronize()
    attn_ms = statistics.mean(evs[s][0][l].elapsed_time(evs[s][1][l]) for s in range(K) for l in range(L))
    st[0] = api.get_status()
    if int(st[0]) != api.SSBA_OK:
        raise RuntimeError(f"device status {int(st[0])} after the timed region")

    F_layer = kept_flops(w.B, w.heads, Tb, keep, w.head_dim)
    value = whole_job_tflops(world, L * F_layer, ms_step * 1e-3)

    # ---- roofline of the dominant kernel (the only one: the fused launch). Its average launch
    #      duration over the timed region is the region's event time over its L * K launches (the
    #      launches run back to back on one stream, overlapping only through programmatic
    #      dependent launch); the duration with an event around each launch, which ends that
    #      overlap, is reported beside it.
    hbm_gbs, bf16_tflops, peak_src = measured_peaks()
    layer_ms = ms_step / L
    attn_tflops = F_layer / (layer_ms * 1e-3) / 1e12
    attn_tflops_ev = F_layer / (attn_ms * 1e-3) / 1e12
    # Q, K, V read and O written once, lse written, the block means written
    attn_bytes = (4 * w.B * w.heads * w.N * w.head_dim * 2 + w.B * w.heads * w.N * 4
                  + 2 * w.B * w.heads * Tb * w.head_dim * 4)
    traffic = profiled_traffic()
    roofline = {"kernel": "ssba_attn_tc_kernel (ssba_forward_fused)", "bound": "tensor", "achieved": attn_tflops,
                "peak": bf16_tflops, "unit": "TFLOP/s", "frac": attn_tflops / bf16_tflops,
                "traffic": traffic, "algorithmic_bytes": attn_bytes,
                "algorithmic_flops": F_layer, "avg_launch_ms": layer_ms,
                "how": "algorithmic flops per launch / (timed-region event time / launches in it)",
                "per_launch_events": {"avg_launch_ms": attn_ms, "achieved": attn_tflops_ev,
                                      "frac": attn_tflops_ev / bf16_tflops,
                                      "how": "an event pair around each launch of K more steps (ends the overlap "
                                             "of consecutive launches)"},
                "peak_source": f"{peak_src} dense bf16 (burst)",
                "frac_of_sustained": attn_tflops / measured_peaks_sustained(),
                "hbm_frac": attn_bytes / (layer_ms * 1e-3) / 1e9 / hbm_gbs}

    # ---- the same layers with the pooling as a launch of its own (ssba_pool_blocks, then
    #      ssba_forward_select), outside the timed region: its step time, and the pooling kernel's
    #      duration (CUDA events around each launch) for its own roofline
    pool_bytes = 2 * w.B * w.heads * w.N * w.head_dim * 2 + 2 * w.B * w.heads * Tb * w.head_dim * 4
    pool_select = None
    mask_roof = None
    mask_ms = None
    try:
        def step_ps():
            for ly in layers:
                ly.pool()
                ly.attend()

        for _ in range(3):
            step_ps()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(5):
            step_ps()
        e1.record(stream)
        torch.cuda.synchronize()
        tps = e0.elapsed_time(e1) / 5
        evp = [[torch.cuda.Event(enable_timing=True) for _ in range(L)] for _ in range(3)]
        for l, ly in enumerate(layers):
            evp[0][l].record(stream)
            ly.pool()
            evp[1][l].record(stream)
            ly.attend()
            evp[2][l].record(stream)
        torch.cuda.synchronize()
        mask_ms = statistics.mean(evp[0][l].elapsed_time(evp[1][l]) for l in range(L))
        sel_ms = statistics.mean(evp[1][l].elapsed_time(evp[2][l]) for l in range(L))
        pool_select = {"ms_per_step": tps, "value": whole_job_tflops(1, L * F_layer, tps * 1e-3),
                       "pool_ms_per_layer": mask_ms, "select_attention_ms_per_layer": sel_ms,
                       "how": "ssba_pool_blocks + ssba_forward_select per layer, CUDA events around 5 steps; "
                              "per-kernel durations from events around each launch of one step"}
        mask_roof = {"kernels": "ssba_pool_blocks_kernel (pool + select path, 1 launch per layer)", "bound": "hbm",
                     "achieved": pool_bytes / (mask_ms * 1e-3) / 1e9, "peak": hbm_gbs, "unit": "GB/s",
                     "frac": pool_bytes / (mask_ms * 1e-3) / 1e9 / hbm_gbs, "algorithmic_bytes": pool_bytes,
                     "avg_call_ms": mask_ms}
    except Exception as exc:  # reported, not fatal
        pool_select = f"failed: {exc}"

    # ---- the two-launch path on the same layers (mask kernel with its selection, then the forward
    #      on the lists), outside the timed region
    two_launch = None
    try:
        def step2():
            for ly in layers2:
                ly.mask()
                ly.attend()

        for _ in range(3):
            step2()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(5):
            step2()
        e1.record(stream)
        torch.cuda.synchronize()
        t2 = e0.elapsed_time(e1) / 5
        two_launch = {"ms_per_step": t2, "value": whole_job_tflops(1, L * F_layer, t2 * 1e-3),
                      "how": "ssba_build_mask + ssba_forward per layer, CUDA events around 5 steps"}
    except Exception as exc:  # reported, not fatal
        two_launch = f"failed: {exc}"

    # ---- dense attention from the same build, same shape (outside the timed region)
    dense_ms = None
    try:
        Od = torch.empty(shp, dtype=w.dtype, device=dev)
        ld = torch.empty(shp[:3], dtype=torch.float32, device=dev)
        for _ in range(3):
            api.forward_dense(descs[0], Qs[0], Ks[0], Vs[0], Od, ld)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = L  # the step's layers, back to back like the sparse step
        e0.record(stream)
        for r in range(reps):
            api.forward_dense(descs[r % 2], Qs[r % L], Ks[r % L], Vs[r % L], Od, ld)
        e1.record(stream)
        torch.cuda.synchronize()
        dense_ms = e0.elapsed_time(e1) / reps
    except Exception as exc:  # reported, not fatal
        dense_ms = f"failed: {exc}"

    # ---- the text segment of Algorithm 1: every image query also attends to 256 text keys
    #      (outside the timed region; the same layers and masks)
    joint = None
    try:
        T_txt = 256
        kv_t = [synthetic.qkv(w.B, w.heads, T_txt, w.head_dim, w.dtype, seed=500 + l + 1000 * rank)[:2]
                for l in range(L)]
        Kts = [a.to(dev) for a, _ in kv_t]
        Vts = [b.to(dev) for _, b in kv_t]
        Oj = torch.empty(shp, dtype=w.dtype, device=dev)
        lj = torch.empty(shp[:3], dtype=torch.float32, device=dev)
        for l in range(3):
            api.forward_joint(descs[l], Qs[l], Ks[l], Vs[l], Kts[l], Vts[l], idx[l], cnt[l], Oj, lj)
        reps = 2 * L
        evj = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for r in range(reps):
            l = r % L
            evj[r][0].record(stream)
            api.forward_joint(descs[l], Qs[l], Ks[l], Vs[l], Kts[l], Vts[l], idx[l], cnt[l], Oj, lj)
            evj[r][1].record(stream)
        torch.cuda.synchronize()
        tj = statistics.mean(a.elapsed_time(b) for a, b in evj)
        F_joint = 4.0 * w.B * w.heads * w.N * (T_txt + keep * 64) * w.head_dim
        joint = {"T_txt": T_txt, "attention_ms_per_layer": tj, "effective_tflops": F_joint / (tj * 1e-3) / 1e12,
                 "flops_per_layer": F_joint,
                 "how": "ssba_forward_joint per layer (text keys first, then the kept image blocks), CUDA events "
                        "around each call, synthetic text K/V"}
    except Exception as exc:  # reported, not fatal
        joint = f"failed: {exc}"

    # ---- the backward pass (gradients over the same kept blocks) of a few layers; outside the
    #      timed region. Algorithmic FLOPs: QK^T, dP = dO V^T, dV, dQ, dK on the kept blocks,
    #      2.5 x the forward's
    bwd = None
    try:
        gos = [synthetic.qkv(w.B, w.heads, w.N, w.head_dim, w.dtype, seed=700 + l + 1000 * rank)[0].to(dev)
               for l in range(2)]
        wsb = torch.empty(api.backward_workspace_bytes(descs[0]), dtype=torch.uint8, device=dev)
        grads = [torch.empty(shp, dtype=torch.float32, device=dev) for _ in range(3)]
        api.backward(descs[0], Qs[0], Ks[0], Vs[0], Os[0], lses[0], gos[0], idx[0], cnt[0], *grads, workspace=wsb)
        reps = 6
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for r in range(reps):
            l = r % 2
            api.backward(descs[l], Qs[l], Ks[l], Vs[l], Os[l], lses[l], gos[l], idx[l], cnt[l], *grads, workspace=wsb)
        e1.record(stream)
        torch.cuda.synchronize()
        tb = e0.elapsed_time(e1) / reps
        F_b = 2.5 * F_layer
        # the same call at 2048 px (rows of 41 kept blocks of 256), one layer with its own mask
        # and forward, outside the timed region
        big = None
        try:
            wb = synthetic.PX2048
            db = api.SsbaDesc(wb.B, wb.heads, wb.H_tok, wb.W_tok, shift_r=4, shift_c=4, rho=wb.rho, dtype=wb.dtype)
            qb_, kb_, vb_ = (t.to(dev) for t in synthetic.qkv(wb.B, wb.heads, wb.N, wb.head_dim, wb.dtype,
                                                               seed=900 + 1000 * rank, std=wb.std))
            gob = synthetic.qkv(wb.B, wb.heads, wb.N, wb.head_dim, wb.dtype, seed=901 + 1000 * rank)[0].to(dev)
            ib, cb = api.build_mask(db, qb_, kb_)
            Ob, lb = api.forward(db, qb_, kb_, vb_, ib, cb)
            wsbb = torch.empty(api.backward_workspace_bytes(db), dtype=torch.uint8, device=dev)
            gb = [torch.empty((wb.B, wb.heads, wb.N, wb.head_dim), dtype=torch.float32, device=dev) for _ in range(3)]
            api.backward(db, qb_, kb_, vb_, Ob, lb, gob, ib, cb, *gb, workspace=wsbb)
            e0.record(stream)
            for _ in range(4):
                api.backward(db, qb_, kb_, vb_, Ob, lb, gob, ib, cb, *gb, workspace=wsbb)
            e1.record(stream)
            torch.cuda.synchronize()
            tbb = e0.elapsed_time(e1) / 4
            keep_b = api.keep_count(db)
            F_bb = 2.5 * kept_flops(wb.B, wb.heads, db.Tb, keep_b, wb.head_dim)
            big = {"config": wb.name, "keep": keep_b, "Tb": db.Tb, "ms_per_layer": tbb,
                   "effective_tflops": F_bb / (tbb * 1e-3) / 1e12, "flops_per_layer": F_bb}
            del qb_, kb_, vb_, gob, Ob, lb, wsbb, gb
        except Exception as exc:  # reported, not fatal
            big = f"failed: {exc}"
        bwd = {"ms_per_layer": tb, "effective_tflops": F_b / (tb * 1e-3) / 1e12, "flops_per_layer": F_b,
               "px2048": big,
               "how": "ssba_backward per layer (a row kernel: D, the rows' (lse, D) by block, the key "
                      "blocks' transposed lists; then the persistent warp-specialised tcgen05 kernel, "
                      "dQ per query block and dK, dV per key block) on the layer's forward O and lse "
                      "and a synthetic dO, CUDA events"}
    except Exception as exc:  # reported, not fatal
        bwd = f"failed: {exc}"

    # ---- one level of the T-DVAE's Haar bank and its inverse on a VAE-sized feature map
    #      (128 channels of 1024 x 1024, bf16; 256 MiB each way, larger than L2); outside the
    #      timed region. Algorithmic bytes: every input element read once, every output written once
    haar = None
    try:
        hN, hC, hH, hW = 1, 128, 1024, 1024
        hx = synthetic.feature_map(hN, hC, hH, hW, torch.bfloat16, seed=900 + rank).to(dev)
        hy = torch.empty((hN, 4 * hC, hH // 2, hW // 2), dtype=torch.bfloat16, device=dev)
        hy3 = torch.empty((hN, 3 * hC, hH // 2, hW // 2), dtype=torch.bfloat16, device=dev)
        hb = torch.empty_like(hx)
        hp = [torch.empty((hN, 4 * hC, hH >> l, hW >> l), dtype=torch.bfloat16, device=dev) for l in (1, 2, 3)]
        nbytes = hx.numel() * 2
        pyr_bytes = nbytes + 4 * sum(nbytes >> (2 * l) for l in (1, 2, 3))  # x once, 4 bands per level
        peak = hbm_gbs
        out = {}
        for name, fn, moved in (("dwt_nb4", lambda: api.haar_dwt(hx, 4, y=hy, stream=stream), 2 * nbytes),
                                ("dwt_nb3", lambda: api.haar_dwt(hx, 3, y=hy3, stream=stream), nbytes * 7 // 4),
                                ("iwt_nb4", lambda: api.haar_iwt(hy, hC, 4, x=hb, stream=stream), 2 * nbytes),
                                ("dwt_pyramid3", lambda: api.haar_dwt_pyramid(hx, 3, 4, ys=hp, stream=stream),
                                 pyr_bytes),
                                ("iwt_pyramid3", lambda: api.haar_iwt_pyramid(hp, hC, 4, x=hb, stream=stream),
                                 nbytes + 3 * sum(nbytes >> (2 * l) for l in (1, 2, 3)) + (nbytes >> 6))):
            for _ in range(3):
                fn()
            reps = 10
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                fn()
            e1.record(stream)
            torch.cuda.synchronize()
            t = e0.elapsed_time(e1) / reps
            gbs = moved / (t * 1e-3) / 1e9
            out[name] = {"us": t * 1e3, "bytes": moved, "achieved_gbs": gbs,
                         "frac": gbs / peak}
        haar = dict(out, shape=[hN, hC, hH, hW], dtype="bf16", peak_gbs=peak, peak_source=peak_src,
                    how="ssba_haar_dwt / ssba_haar_iwt (one level) and the 3-level pyramids, back to back, "
                        "CUDA events around 10 launches; bytes: each input element read once, each output "
                        "element written once (the inverse pyramid reads LL of level 3 and the detail "
                        "bands); frac of the HBM copy bandwidth")
        del hx, hy, hy3, hb, hp
    except Exception as exc:  # reported, not fatal
        haar = f"failed: {exc}"

    def events_ms(fn, reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    # ---- layer-aware sparsity: the same 24 layers with the synthetic per-layer schedule
    #      (edge layers at 75 %, the middle sparser, 84.16 % on average); outside the timed region
    layer_aware = None
    try:
        from paper_2605_15684_gb300 import schedule
        rhos = schedule.layer_rhos(L, Tb)
        ldescs = [api.SsbaDesc(w.B, w.heads, w.H_tok, w.W_tok, w.head_dim, 8, *layer_shift(l), rhos[l], w.dtype)
                  for l in range(L)]
        lkeep = [api.keep_count(d) for d in ldescs]
        lidx = [torch.empty((w.B, w.heads, Tb, k), dtype=torch.int32, device=dev) for k in lkeep]
        llayers = [api.BoundSelectLayer(ldescs[l], Qs[l], Ks[l], Vs[l], qbs[l], kbs[l], lidx[l], cnt[l], Os[l],
                                        lses[l], stream) for l in range(L)]

        def lstep():
            for ly in llayers:
                ly.fused()

        for _ in range(3):
            lstep()
        tl = events_ms(lstep, 5)
        F_l = sum(kept_flops(w.B, w.heads, Tb, k, w.head_dim) for k in lkeep)
        layer_aware = {"ms_per_step": tl, "effective_tflops": F_l / (tl * 1e-3) / 1e12,
                       "mean_sparsity": 1.0 - sum(lkeep) / (L * Tb), "keep_per_layer": lkeep,
                       "uniform_ms_per_step": ms_step,
                       "how": "the fused launch (ssba_forward_fused) of the 24 layers with rho_l from "
                              "schedule.layer_rhos, CUDA events around 5 steps"}
    except Exception as exc:  # reported, not fatal
        layer_aware = f"failed: {exc}"

    # ---- the other workloads of the paper's range, outside the timed region: the 512 px model
    #      (24 layers), the elastic sweep at 1024 px (32x32 and 64x64 grids x sparsity x batch)
    #      and the 2048 px stress (24 layers, 84 % and 90 %). Per config: the time per layer on
    #      its path (the fused launch for Tb <= 256, else ssba_build_mask + ssba_forward), the
    #      effective TFLOP/s over kept blocks and its fraction of the measured peak, and the
    #      same-build dense kernel. Inputs: N(0,1) (512 px: x 1/8) drawn on the device from a
    #      seeded generator, alternating shifts, and enough distinct layers that one pass over
    #      them is larger than L2 (cold inputs per layer, as in the timed step)
    sweep = None
    try:
        def run_config(Bc, Hc, Wc, rho, std, layers):
            Tbc = Hc * Wc // 64
            dsc = [api.SsbaDesc(Bc, w.heads, Hc, Wc, w.head_dim, 8, *layer_shift(l), rho, w.dtype)
                   for l in range(layers)]
            kc = api.keep_count(dsc[0])
            shp_c = (Bc, w.heads, Hc * Wc, w.head_dim)
            gen = torch.Generator(device=dev)
            gen.manual_seed(4000 + 1000 * rank)
            ins = [[(torch.randn(shp_c, generator=gen, device=dev) * std).to(w.dtype) for _ in range(3)]
                   for _ in range(layers)]
            Oc = torch.empty(shp_c, dtype=w.dtype, device=dev)
            lc = torch.empty(shp_c[:3], dtype=torch.float32, device=dev)
            ic = torch.empty((Bc, w.heads, Tbc, kc), dtype=torch.int32, device=dev)
            cc = torch.empty((Bc, w.heads, Tbc), dtype=torch.int32, device=dev)
            if Tbc <= 256:
                pq = torch.empty((Bc, w.heads, Tbc, w.head_dim), dtype=torch.float32, device=dev)
                pk = torch.empty_like(pq)
                lys = [api.BoundSelectLayer(dsc[l], *ins[l], pq, pk, ic, cc, Oc, lc, stream) for l in range(layers)]

                def fn():
                    for ly in lys:
                        ly.fused()
                path = "ssba_forward_fused"
                # the two calls of the API (mask kernel, then the forward on its lists), timed the same way
                wsc = torch.empty(api.mask_workspace_bytes(dsc[0]), dtype=torch.uint8, device=dev)
                lys2 = [api.BoundLayer(dsc[l], *ins[l], ic, cc, Oc, lc, wsc, stream) for l in range(layers)]

                def fn2():
                    for ly in lys2:
                        ly.mask()
                        ly.attend()
                for _ in range(3):
                    fn2()
                t_two = events_ms(fn2, 5) / layers
            else:
                wsc = torch.empty(api.mask_workspace_bytes(dsc[0]), dtype=torch.uint8, device=dev)
                lys = [api.BoundLayer(dsc[l], *ins[l], ic, cc, Oc, lc, wsc, stream) for l in range(layers)]

                def fn():
                    for ly in lys:
                        ly.mask()
                        ly.attend()
                path = "ssba_build_mask + ssba_forward"
            for _ in range(3):
                fn()
            t_layer = events_ms(fn, 5) / layers
            nd = min(layers, 8)

            def fd():
                for l in range(nd):
                    api.forward_dense(dsc[l], *ins[l], Oc, lc)
            fd()
            t_dense = events_ms(fd, 3) / nd
            Fc = kept_flops(Bc, w.heads, Tbc, kc, w.head_dim)
            tf = Fc / (t_layer * 1e-3) / 1e12
            del ins, lys
            out = {"grid": [Hc, Wc], "B": Bc, "rho": rho, "keep": kc, "Tb": Tbc,
                    "realized_sparsity": round((Tbc - kc) / Tbc, 6), "layers": layers, "path": path,
                    "ms_per_layer": t_layer, "effective_tflops": tf, "frac": tf / bf16_tflops,
                    "dense_ms_per_layer": t_dense, "speedup_vs_dense": t_dense / t_layer,
                    "ideal_speedup_vs_dense": Tbc / kc}
            if Tbc <= 256:
                out["two_call_ms_per_layer"] = t_two  # ssba_build_mask + ssba_forward
            return out

        def n_layers(Bc, Hc, Wc):
            per = 3 * Bc * w.heads * Hc * Wc * w.head_dim * 2
            return min(24, max(1, math.ceil(2 * 129e6 / per)))

        cases = {"512px_24_layers": run_config(1, 32, 32, 0.8416, 0.125, 24)}
        for (Hc, Wc) in ((32, 32), (64, 64)):
            for Bc in (1, 4):
                for rho in (0.0, 0.5, 0.75, 0.8416, 0.9):
                    cases[f"sweep_{Hc}x{Wc}_B{Bc}_rho{rho}"] = run_config(Bc, Hc, Wc, rho, 1.0, n_layers(Bc, Hc, Wc))
        for rho in (0.84, 0.9):
            cases[f"2048px_24_layers_rho{rho}"] = run_config(1, 128, 128, rho, 1.0, 24)
        # the headline layer back to back on resident inputs (warm L2) against the timed step (cold)
        warm = events_ms(lambda: layers[1].fused(), 20)
        cases["1024px_warm_l2"] = {"ms_per_layer": warm, "effective_tflops": F_layer / (warm * 1e-3) / 1e12,
                                   "how": "one shifted 1024 px layer's fused launch 20 times back to back"}
        sweep = dict(cases, peak_tflops=bf16_tflops, peak_source=peak_src,
                     how="CUDA events around 5 passes over the config's layers after 3 warm-up passes; "
                         "dense: ssba_forward_dense on up to 8 of the layers; two_call_ms_per_layer: "
                         "ssba_build_mask then ssba_forward per layer, timed the same way")
    except Exception as exc:  # reported, not fatal
        sweep = f"failed: {exc}"

    # ---- the steps before the mask fused into the projection (ssba_qkv_rope_pool): X W^T + b, RoPE,
    #      block means; 1024 px, Dm = 1536; X and Wqkv (27 MB) stay in L2 between launches
    qkv = None
    try:
        Dm = w.heads * w.head_dim
        X, Wq, bq = (t.to(dev) for t in synthetic.projection_inputs(w.B, w.N, Dm, seed=800 + rank))
        pshp = (w.B, w.heads, Tb, w.head_dim)
        outs = [torch.empty(shp, dtype=torch.bfloat16, device=dev) for _ in range(3)] + \
               [torch.empty(pshp, dtype=torch.float32, device=dev) for _ in range(2)]
        flops_qkv = 2.0 * w.B * w.N * Dm * 3 * Dm
        qkv = {"flops": flops_qkv, "peak_tflops": bf16_tflops, "peak_source": peak_src}
        for name, sh in (("unshifted", (0, 0)), ("shifted", (4, 4))):
            dq = api.SsbaDesc(w.B, w.heads, w.H_tok, w.W_tok, w.head_dim, 8, *sh, w.rho, w.dtype)
            fn = (lambda dq=dq: api.qkv_rope_pool(dq, X, Wq, bq, out=outs, stream=stream))
            for _ in range(3):
                fn()
            tq = events_ms(fn, 20)
            qkv[name] = {"us": tq * 1e3, "tflops": flops_qkv / (tq * 1e-3) / 1e12,
                         "frac": flops_qkv / (tq * 1e-3) / 1e12 / bf16_tflops}
        lin = (lambda: torch.nn.functional.linear(X, Wq))
        for _ in range(3):
            lin()
        tc = events_ms(lin, 20)
        qkv["cublas_plain_projection"] = {"us": tc * 1e3, "tflops": flops_qkv / (tc * 1e-3) / 1e12}
        qkv["how"] = ("ssba_qkv_rope_pool (tcgen05, bias + 2-D RoPE + block means fused) against "
                      "torch.nn.functional.linear (cuBLAS, the bare X W^T); CUDA events around 20 launches")
    except Exception as exc:  # reported, not fatal
        qkv = f"failed: {exc}"

    # ---- end to end through the public API with host buffers (pinned), copies timed
    e2e = None
    if args.e2e_steps > 0:
        pin = [[t.pin_memory() for t in h] for h in host_qkv]
        O_h = [torch.empty(shp, dtype=w.dtype).pin_memory() for _ in range(L)]
        l_h = [torch.empty(shp[:3], dtype=torch.float32).pin_memory() for _ in range(L)]
        h2d_s = torch.cuda.Stream(device=dev)
        d2h_s = torch.cuda.Stream(device=dev)
        h2d_done = [torch.cuda.Event() for _ in range(L)]
        comp_done = [torch.cuda.Event() for _ in range(L)]
        d2h_done = [torch.cuda.Event() for _ in range(L)]

        def e2e_step():
            for l in range(L):
                h2d_s.wait_event(comp_done[l])  # previous step's layer l no longer reads its inputs
                with torch.cuda.stream(h2d_s):
                    Qs[l].copy_(pin[l][0], non_blocking=True)
                    Ks[l].copy_(pin[l][1], non_blocking=True)
                    Vs[l].copy_(pin[l][2], non_blocking=True)
                h2d_done[l].record(h2d_s)
            for l, ly in enumerate(layers):
                stream.wait_event(h2d_done[l])
                stream.wait_event(d2h_done[l])  # previous step's read-back of O[l] finished
                ly.fused()
                comp_done[l].record(stream)
                d2h_s.wait_event(comp_done[l])
                with torch.cuda.stream(d2h_s):
                    O_h[l].copy_(Os[l], non_blocking=True)
                    l_h[l].copy_(lses[l], non_blocking=True)
                d2h_done[l].record(d2h_s)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step()
        torch.cuda.synchronize()
        e2e_s = (time.perf_counter() - t0) / args.e2e_steps
        e2e_s = max_over_ranks(e2e_s, world, dev)
        h2d = L * 3 * w.B * w.heads * w.N * w.head_dim * 2
        d2h = L * (w.B * w.heads * w.N * w.head_dim * 2 + w.B * w.heads * w.N * 4)
        e2e = {"value": whole_job_tflops(world, L * F_layer, e2e_s), "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_s * 1e3, "steps": args.e2e_steps,
               "how": "pinned host Q/K/V -> device on a copy stream, the fused launch (ssba_forward_fused), O and "
                      "lse -> pinned host on a second copy stream; host wall clock around the steps"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        threads = oracle.max_threads()
        heads_sample = max(1, min(w.heads, threads))
        rate, dt = oracle_sample(w, heads_sample)
        cpu = {"value": rate, "unit": "TFLOP/s", "cores": min(threads, heads_sample), "kind": "oracle",
               "nproc": os.cpu_count(), "cpu_model": cpu_model(),
               "sample": f"{heads_sample} of {w.heads} heads of one layer (mask + forward), {dt:.2f} s, "
                         f"fp64 C with OpenMP over heads"}
        try:  # one thread at the 512 px config
            from paper_2605_15684_gb300 import synthetic as _syn
            oracle.set_threads(1)
            rate1, dt1 = oracle_sample(_syn.PX512, 8)
            cpu["single_thread_512px"] = {"value": rate1, "unit": "TFLOP/s", "cores": 1, "seconds": dt1,
                                          "sample": "8 of 24 heads of one 512 px layer (mask + forward)"}
        except Exception as exc:  # reported, not fatal
            cpu["single_thread_512px"] = f"failed: {exc}"
        finally:
            oracle.set_threads(threads)

    # ---- the mask when the projection has pooled: selection alone (ssba_select_mask) against the
    #      full build (ssba_build_mask re-reads Q and K); 20 launches captured in a CUDA graph,
    #      since one launch is shorter than its host call
    mask_split = None
    if isinstance(qkv, dict):
        try:
            d1 = descs[1]
            qb_, kb_ = outs[3], outs[4]
            sidx = torch.empty((w.B, w.heads, Tb, keep), dtype=torch.int32, device=dev)
            scnt = torch.empty((w.B, w.heads, Tb), dtype=torch.int32, device=dev)
            res = {}
            for name, fn in (("select_from_pooled", lambda: api.select_mask(d1, qb_, kb_, sidx, scnt)),
                             ("full_mask_build",
                              lambda: api.build_mask(d1, Qs[1], Ks[1], sidx, scnt, workspace=ws))):
                fn()
                torch.cuda.synchronize()
                graph = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graph):
                    for _ in range(20):
                        fn()
                graph.replay()
                torch.cuda.synchronize()
                res[name + "_us"] = events_ms(graph.replay, 5) / 20 * 1e3
            mask_split = dict(res, how="per launch, 20 launches per CUDA graph, 5 replays, 1024 px layer")
        except Exception as exc:  # reported, not fatal
            mask_split = f"failed: {exc}"

    # ---- the mask kernel against the HBM roofline: ssba_build_mask (one ssba_mask_fused_kernel
    #      launch) over the step's layers, each with its own Q and K (larger than L2 together),
    #      captured in a CUDA graph; algorithmic bytes = Q + K read once
    mask_roofline = None
    try:
        midx = torch.empty((w.B, w.heads, Tb, keep), dtype=torch.int32, device=dev)
        mcnt = torch.empty((w.B, w.heads, Tb), dtype=torch.int32, device=dev)
        api.build_mask(descs[0], Qs[0], Ks[0], midx, mcnt, workspace=ws)
        torch.cuda.synchronize()
        mgraph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(mgraph):
            for l in range(L):
                api.build_mask(descs[l], Qs[l], Ks[l], midx, mcnt, workspace=ws)
        mgraph.replay()
        torch.cuda.synchronize()
        m_us = events_ms(mgraph.replay, 5) / L * 1e3
        m_bytes = 2 * w.B * w.heads * w.N * w.head_dim * 2
        m_ach = m_bytes / (m_us * 1e-6) / 1e9
        mask_roofline = {"kernel": "ssba_mask_fused_kernel (ssba_build_mask)", "bound": "hbm",
                         "achieved": m_ach, "peak": hbm_gbs, "unit": "GB/s", "frac": m_ach / hbm_gbs,
                         "traffic": profiled_traffic(MASK_PROFILE, MASK_SOURCES),
                         "us_per_layer": m_us, "algorithmic_bytes": m_bytes,
                         "how": "one launch per layer over the step's layers (distinct Q, K: larger than "
                                "L2), captured in a CUDA graph, 5 replays; Q + K read once per launch"}
        assert api.get_status() == api.SSBA_OK
    except Exception as exc:  # reported, not fatal
        mask_roofline = f"failed: {exc}"

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": K,
            "warmup": max(3, args.warmup), "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": dict(config_dict(w, keep, L), parallelism="replicas" if world > 1 else "single GPU"),
            "latency_ms_per_layer": ms_step / L,
            "attention_ms_per_layer": attn_ms,
            "roofline": roofline, "roofline_pool": mask_roof,
            "pool_select_path": pool_select,
            "two_launch_path": two_launch,
            "dense_attention_ms_per_layer": dense_ms,
            "text_joint": joint,
            "backward": bwd,
            "haar": haar,
            "layer_aware": layer_aware,
            "configs_sweep": sweep,
            "qkv_fused": qkv,
            "mask_after_fused_pooling": mask_split,
            "roofline_mask": mask_roofline,
            "speedup_vs_dense": (dense_ms / layer_ms) if isinstance(dense_ms, float) else None,
            "speedup_vs_dense_how": "per layer, both back to back over the step's layers: "
                                    "ssba_forward_dense against the fused sparse launch",
            "ideal_speedup_vs_dense": Tb / keep,
            "e2e": e2e, "cpu_baseline": cpu,
            "gpu_launches": K * L,
            "clocks": clocks.summary(wall0, wall1),
        }
        print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        torch.distributed.init_process_group("nccl")
    try:
        run_ours(args, rank, world)
    finally:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
