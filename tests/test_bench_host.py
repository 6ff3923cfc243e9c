"""Host-side pieces of the benchmark: the algorithmic work it counts for the
roofline (window points and edge-bins, from the +-k sigma windows), the measured
peak it reads, and the committed profile's traffic line."""
import math
import os

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import bench  # noqa: E402


def test_algorithmic_work_counts_window_bins():
    rng = np.random.default_rng(3)
    V, B, D, k = 7, 5, 20, 6.0
    mu = rng.uniform(-5, D + 5, size=(V, B)).astype(np.float32)
    sg = rng.uniform(0.05, 3.0, size=(V, B)).astype(np.float32)
    src = np.array([0, 0, 1, 2, 3, 5], np.int64)
    dst = np.array([1, 2, 3, 4, 6, 6], np.int64)
    flops, n_pt, n_eb = bench.algorithmic_flops(torch, torch.from_numpy(mu), torch.from_numpy(sg),
                                                torch.from_numpy(src), torch.from_numpy(dst), k, D)
    # brute force: the points t with |t + 1/2 - mu| <= k sigma, clipped to [0, D - 2];
    # a window of n points covers n + 1 bins
    bins = np.zeros((V, B))
    for v in range(V):
        for b in range(B):
            pts = [t for t in range(0, D - 1) if abs(t + 0.5 - float(mu[v, b])) <= k * float(sg[v, b])]
            bins[v, b] = len(pts) + 1
    assert n_pt == pytest.approx(bins.sum())
    assert n_eb == pytest.approx(sum((2 * bins[u] + bins[w]).sum() for u, w in zip(src, dst)))
    assert flops == pytest.approx(20 * n_pt + 8 * n_eb)


def test_measured_hbm_peak_is_read_or_falls_back():
    v = bench.measured_hbm_gbs()
    assert 1000.0 < v < 20000.0


def test_profiled_traffic_is_a_byte_count_or_none():
    t = bench.profiled_traffic()
    assert t is None or (math.isfinite(t) and 1e6 < t < 1e10)
