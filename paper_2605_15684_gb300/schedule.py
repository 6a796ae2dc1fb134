"""Layer-aware sparsity (Sec. 2.2 "layer-importance-aware execution"; Table 2: 84.16 %
average sparsity against 75 % uniform). The paper gives only the average, not the per-layer
ratios, so this schedule is synthetic: the first and last layers keep the uniform ratio, and
the drop count rises linearly towards the middle layers, with integer drop counts fitted so
that the mean dropped fraction over the layers is the target. No arithmetic of the attention
itself lives here; the ratios go into each layer's descriptor."""
from __future__ import annotations


def layer_drop_counts(layers: int, Tb: int, target: float = 0.8416, edge: float = 0.75) -> list[int]:
    """Integer drop counts k_l (k = floor(Tb * rho_l) of Algorithm 1), edge layers at
    floor(Tb * edge), a triangle in between, sum as close as possible to target * Tb * layers,
    every layer keeping at least one block. One or two layers take the target uniformly."""
    if layers < 1 or Tb < 2:
        raise ValueError("need at least one layer and two blocks")
    k_max = Tb - 1
    want = round(target * Tb * layers)
    if layers <= 2:  # no middle layers: uniform at the target
        return [min(k_max, round(target * Tb))] * layers
    k_edge = int(Tb * edge)
    tri = [1.0 - abs(2.0 * l / (layers - 1) - 1.0) for l in range(layers)]

    def counts(a: float) -> list[int]:
        return [min(k_max, k_edge + int(round(a * t))) for t in tri]

    lo, hi = 0.0, float(Tb)
    for _ in range(60):  # bisection on the triangle's height
        mid = 0.5 * (lo + hi)
        if sum(counts(mid)) < want:
            lo = mid
        else:
            hi = mid
    best = min((counts(lo), counts(hi)), key=lambda c: abs(sum(c) - want))
    # close the last few blocks of the gap one layer at a time, middle layers first
    order = sorted(range(layers), key=lambda l: -tri[l])
    gap = want - sum(best)
    for l in order:
        if gap == 0:
            break
        step = 1 if gap > 0 else -1
        if k_edge <= best[l] + step <= k_max and tri[l] > 0:
            best[l] += step
            gap -= step
    return best


def layer_rhos(layers: int, Tb: int, target: float = 0.8416, edge: float = 0.75) -> list[float]:
    """Sparse ratios rho_l whose floor(Tb * rho_l) is exactly layer_drop_counts (half a block
    of margin against rounding)."""
    return [(k + 0.5) / Tb for k in layer_drop_counts(layers, Tb, target, edge)]
