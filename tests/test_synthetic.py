"""The seeded workload generator: shapes, packing and recipes (no GPU)."""
import numpy as np
import pytest

from paper_2607_07508_gb300 import synthetic as S


@pytest.mark.parametrize("name", S.CONFIG_NAMES)
def test_config_shapes_and_packing(name):
    wl = S.make_workload(name, dense=False)
    cu = wl.cu_seqlens
    assert cu.dtype == np.int32 and cu[0] == 0 and cu[-1] == wl.N
    assert np.all(np.diff(cu) >= 0)
    assert len(cu) == wl.B + 1
    for a in (wl.loss_mask, wl.values, wl.y, wl.xi, wl.logp_syn):
        assert len(a) == wl.N
    assert len(wl.rewards) == wl.B
    assert wl.y.min() >= 0 and wl.y.max() < wl.V
    assert set(np.unique(wl.rewards)) <= {0.0, 1.0}
    want_N = {"small": 98304, "moe": 65536, "long": 524288, "large": 262144}
    if name in want_N:
        assert wl.N == want_N[name]


def test_config_recipes():
    moe = S.make_workload("moe", dense=False)
    obs = 1.0 - moe.loss_mask.mean()
    assert 0.15 < obs < 0.35 and moe.lam == 0.95 and (moe.eps_low, moe.eps_high) == (0.3, 5.0)
    lng = S.make_workload("long", dense=False)
    L = np.diff(lng.cu_seqlens)
    assert lng.B == 16 and L.min() >= 16384 and L.max() <= 131072
    assert 0.3 < 1.0 - lng.loss_mask.mean() < 0.55 and lng.alpha == 1.5
    big = S.make_workload("large", dense=False)
    r = np.exp(-big.xi.astype(np.float64))
    out = (r <= 1 - big.eps_low) | (r >= 1 + big.eps_high)
    assert 0.08 < out.mean() < 0.12


def test_determinism():
    a = S.make_workload("tiny")
    b = S.make_workload("tiny")
    assert np.array_equal(a.y, b.y) and np.array_equal(a.values, b.values)
    assert bool((a.H == b.H).all()) and bool((a.W == b.W).all())
