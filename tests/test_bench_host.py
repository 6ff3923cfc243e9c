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


def test_storage_point_edges_pair_consumer_points_with_producers():
    rng = np.random.default_rng(5)
    V, B, D, k = 6, 3, 25, 6.0
    mu = rng.uniform(0, D, size=(V, B)).astype(np.float32)
    sg = rng.uniform(0.1, 2.0, size=(V, B)).astype(np.float32)
    src = np.array([0, 0, 1, 3, 4], np.int64)
    dst = np.array([1, 2, 3, 5, 5], np.int64)
    T = torch.from_numpy
    f, n_pt, n_eb, n_st = bench.algorithmic_work(torch, T(mu), T(sg), T(src), T(dst), k, D, storage=True)
    pts = np.zeros((V, B))
    for v in range(V):
        for b in range(B):
            pts[v, b] = sum(1 for t in range(0, D - 1) if abs(t + 0.5 - float(mu[v, b])) <= k * float(sg[v, b]))
    assert n_st == pytest.approx(sum(pts[w].sum() for w in dst))
    assert f == pytest.approx(20 * n_pt + 8 * (n_eb + n_st))
    _, _, _, none = bench.algorithmic_work(torch, T(mu), T(sg), T(src), T(dst), k, D, storage=False)
    assert none == 0.0


@pytest.mark.parametrize("factor", [1.0, 1.5])
def test_modulo_list_schedule_is_a_verified_witness(factor):
    import oracle
    import workloads as W
    p = W.modulo_loop(3, ii_factor=factor, V=600, levels=20, n_back=30)
    s = bench.modulo_list_schedule(p)
    assert s is not None and s.dtype == np.int32 and s.shape == (p.V,)
    r = oracle.verify(oracle.OracleProblem(p), s)
    assert r["feasible"] == 1 and r["res_ok"] == 1


def test_modulo_list_schedule_gives_up_without_room():
    import workloads as W
    p = W.modulo_loop(3, ii_factor=1.0, V=600, levels=20, n_back=30)
    p.limit = np.where(np.isfinite(p.limit), 0.0, p.limit)   # no slot for any node
    assert bench.modulo_list_schedule(p) is None


def test_launch_count_per_step():
    fused = {"fused": 1, "fused_launches_per_call": 1, "launches_per_iteration": 0}
    multi = {"fused": 0, "fused_launches_per_call": 0, "launches_per_iteration": 8}
    # 20 calls of 100 iterations: one k_fused launch per call, or 8 kernels per
    # iteration, plus legalize and the verifier's two passes per call
    assert bench.launches_per_step(fused, 2000, 100) == 20 * (1 + 3)
    assert bench.launches_per_step(multi, 2000, 100) == 20 * (800 + 3)
    # the path chosen per call: 6 calls on the multi-kernel path (5 kernels per
    # iteration), 14 fused calls, 20 window reductions of the choice
    both = {"fused": 1, "fused_launches_per_call": 1, "launches_per_iteration": 5}
    assert bench.launches_per_step(both, 2000, 100, 14, 600, 20) == 14 + 600 * 5 + 20 + 20 * 3
