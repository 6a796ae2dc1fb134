"""The synthetic layer-aware sparsity schedule: its realised mean drop fraction, its edges and
its shape, checked against the sparsity rule of the oracle (k = floor(Tb * rho))."""
import pytest

import oracle
from paper_2605_15684_gb300 import schedule


@pytest.mark.parametrize("layers,Tb", [(24, 64), (24, 16), (24, 256), (12, 64), (2, 64), (1, 64)])
def test_schedule_mean_edges_and_shape(layers, Tb):
    ks = schedule.layer_drop_counts(layers, Tb)
    rhos = schedule.layer_rhos(layers, Tb)
    # the oracle's sparsity rule gives back exactly the fitted drop counts
    assert [oracle.drop_count(Tb, r) for r in rhos] == ks
    mean = sum(ks) / (layers * Tb)
    assert abs(mean - 0.8416) <= 0.5 / (layers * Tb) + (1.0 / Tb if layers <= 2 else 0.0)
    assert all(oracle.keep_count(Tb, r) >= 1 for r in rhos)
    if layers > 2:
        assert ks[0] == ks[-1] == int(Tb * 0.75)
        mid = layers // 2
        assert all(ks[i] <= ks[i + 1] for i in range(mid - 1))
        assert all(ks[i] >= ks[i + 1] for i in range(mid, layers - 1))


def test_schedule_rejects_degenerate_inputs():
    with pytest.raises(ValueError):
        schedule.layer_drop_counts(0, 64)
    with pytest.raises(ValueError):
        schedule.layer_drop_counts(4, 1)
