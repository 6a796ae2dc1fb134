"""Where the time of one SSBA layer goes: the phases of the fused launch and the tile loop of
its pipelines, from the time stamps of the timeline build (build.py variant "timeline",
-DSSBA_TIMELINE; the default library records nothing).

    python -m paper_2605_15684_gb300.timeline [--layers 24] [--isolated] [--phases-only] [--px 1024]

Runs the benchmark's 1024 px step (64 x 64 grid, B = 1, 24 heads x 64, rho = 0.8416, layer l
with seed l and shift (0,0) / (4,4) alternating, one ssba_forward_fused launch per layer; with
--px 512 or 2048 the 32 x 32 or 128 x 128 grid of those workloads) a few times, then reads the stamps of the last launch (layer 23 in the stream, or, with --isolated,
one more launch of layer 1 alone) and prints:
  * per phase, the min / median / max over the CTAs of globaltimer microseconds since the first
    CTA's entry (pooling copies landed, means stored, grid barrier, staging, selection,
    pipelines start and end);
  * per sampled pipeline, the tile period (SM cycles between the softmax seeing S of
    consecutive tiles) and the median latency of each hand-off in the tile loop.
A diagnostic: the numbers come from a build whose kernels carry extra stores, so read
differences, not absolute times, and time the default build with bench.py.
"""
from __future__ import annotations

import argparse
import ctypes
import statistics

import torch

from . import api, build, synthetic

CTA_EVENTS = ["entry", "dep wait over", "pool rows landed", "means stored", "grid barrier passed",
              "head means staged", "lists selected", "pipelines start", "pipeline 0 done", "pipeline 1 done",
              "exit", "warp 0 selects", "its score row done", "its list done"]
TILE_EVENTS = ["K issued", "QK issued", "softmax saw S", "exps done", "P stored", "PV issued", "V issued",
               "S buffer free", "S loaded", "row max known", "P buffer free", "PV waits over"]
N_CTA, CTA_EV, N_PIPE, N_TILE, TILE_EV, N_ITEM, ITEM_EV = 256, 16, 8, 128, 12, 32, 4


def _read(lib):
    cta = (ctypes.c_uint64 * (N_CTA * CTA_EV))()
    tile = (ctypes.c_uint32 * (N_PIPE * N_TILE * TILE_EV))()
    item = (ctypes.c_uint32 * (N_PIPE * N_ITEM * ITEM_EV))()
    api._raise_on(lib.ssba_timeline_read(cta, tile, item))
    return cta, tile, item


def report(lib, grid: int, tag: str) -> None:
    cta, tile, item = _read(lib)
    rows = [[cta[b * CTA_EV + e] for e in range(CTA_EV)] for b in range(min(grid, N_CTA))]
    t0 = min(r[0] for r in rows if r[0])
    print(f"== {tag}: phases, microseconds since the first CTA's entry (min / median / max over {len(rows)} CTAs)")
    for e, name in enumerate(CTA_EVENTS):
        v = [(r[e] - t0) / 1e3 for r in rows if r[e] >= t0 and r[e]]
        if v:
            print(f"   {name:22s} {min(v):8.2f} {statistics.median(v):8.2f} {max(v):8.2f}")
    print(f"== {tag}: tile loop of the sampled pipelines (SM cycles, medians over tiles)")
    hand = [("QK issued -> softmax saw S", 1, 2), ("saw S -> S loaded", 2, 8), ("S loaded -> max known", 8, 9),
            ("max known -> exps done", 9, 3), ("exps done -> P buffer free", 3, 10), ("P buffer free -> P stored", 10, 4),
            ("P stored -> next saw S", 4, -1),
            ("P stored -> PV waits over", 4, 11), ("PV waits over -> PV issued", 11, 5),
            ("K issued -> QK issued", 0, 1),
            ("S buffer free -> QK issued", 7, 1)]
    for pi in range(N_PIPE):
        def ev(t, e):
            return tile[(pi * N_TILE + t) * TILE_EV + e]
        n = 0
        while n < N_TILE and ev(n, 2) != 0:
            n += 1
        if n < 4:
            continue
        per = [(ev(t + 1, 2) - ev(t, 2)) & 0xFFFFFFFF for t in range(n - 1)]
        line = f"   pipe {pi}: {n} tiles, period med {statistics.median(per):6.0f} (min {min(per)}, max {max(per)})"
        for name, a, b in hand:
            if b < 0:  # the next tile's first event
                d = [(ev(t + 1, 2) - ev(t, a)) & 0xFFFFFFFF for t in range(n - 1) if ev(t, a)]
            else:
                d = [(ev(t, b) - ev(t, a)) & 0xFFFFFFFF for t in range(n) if ev(t, a) and ev(t, b)]
            d = [x for x in d if x < 1 << 30]
            if d:
                line += f"; {name} {statistics.median(d):.0f}"
        print(line)
        start = item[(pi * N_ITEM) * ITEM_EV + 3]
        epi = []
        for k in range(N_ITEM):
            s, o, dn = (item[(pi * N_ITEM + k) * ITEM_EV + e] for e in range(3))
            if o and dn:
                epi.append(((o - start) & 0xFFFFFFFF, (dn - o) & 0xFFFFFFFF))
        if epi:
            print("      items: O ready at " + ", ".join(f"{a}" for a, _ in epi) +
                  "; epilogue " + ", ".join(f"{b}" for _, b in epi) + " cycles")


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--layers", type=int, default=24)
    ap.add_argument("--isolated", action="store_true")
    ap.add_argument("--px", type=int, default=1024, choices=(512, 1024, 2048))
    ap.add_argument("--phases-only", action="store_true",
                    help="the build that records the phase stamps only (per-tile stamps cost time)")
    args = ap.parse_args()
    lib = api.load_library(build.build(variant="phases" if args.phases_only else "timeline"))
    dev = torch.device("cuda", 0)
    w = {512: synthetic.PX512, 1024: synthetic.PX1024, 2048: synthetic.PX2048}[args.px]
    L = args.layers
    descs = [api.SsbaDesc(w.B, w.heads, w.H_tok, w.W_tok, shift_r=4 * (l % 2), shift_c=4 * (l % 2), rho=w.rho,
                          dtype=w.dtype) for l in range(L)]
    keep = api.keep_count(descs[0])
    Tb = descs[0].Tb
    shp = (w.B, w.heads, w.N, w.head_dim)

    def mk(s, dt):
        return torch.empty(s, dtype=dt, device=dev)

    layers = []
    for l in range(L):
        q, k, v = (t.to(dev) for t in synthetic.qkv(w.B, w.heads, w.N, w.head_dim, w.dtype, seed=l, std=w.std))
        layers.append(api.BoundSelectLayer(descs[l], q, k, v, mk((w.B, w.heads, Tb, 64), torch.float32),
                                           mk((w.B, w.heads, Tb, 64), torch.float32),
                                           mk((w.B, w.heads, Tb, keep), torch.int32),
                                           mk((w.B, w.heads, Tb), torch.int32), mk(shp, torch.bfloat16),
                                           mk(shp[:3], torch.float32), torch.cuda.current_stream()))
    for _ in range(3):
        for ly in layers:
            ly.fused()
    torch.cuda.synchronize()
    grid = min(torch.cuda.get_device_properties(dev).multi_processor_count, w.B * w.heads * Tb // 2)
    report(lib, grid, f"layer {L - 1} of a {L}-layer step (in the stream)")
    if args.isolated:
        layers[1].fused()
        torch.cuda.synchronize()
        report(lib, grid, "layer 1 alone")
    assert api.get_status() == api.SSBA_OK


if __name__ == "__main__":
    main()
