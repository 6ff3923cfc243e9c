"""The seeded synthetic workloads have the shapes their recipes state (the inputs
that stand in for the paper's benchmark suites): sizes, degrees, class mixes,
limits, latencies, horizons and back edges."""
import math

import networkx as nx
import numpy as np
import pytest

import workloads as W


def _indeg(p):
    return np.bincount(p.dst, minlength=p.V)


def _outdeg(p):
    return np.bincount(p.src, minlength=p.V)


def _check_dag_and_horizon(p, factor):
    g = nx.DiGraph()
    g.add_nodes_from(range(p.V))
    g.add_edges_from(zip(p.src.tolist(), p.dst.tolist()))
    assert nx.is_directed_acyclic_graph(g)
    assert len(set(zip(p.src.tolist(), p.dst.tolist()))) == p.E      # no duplicate edges
    assert p.cp == int(np.max(p.start + p.lat))
    if factor is not None:
        assert p.D == math.ceil(factor * p.cp)


def test_tiny_layered():
    p = W.tiny_layered(1)
    assert p.V == 64 and p.C == 2 and list(p.limit) == [2, 3]
    assert set(np.unique(p.lat)) <= {1, 2, 3}
    d = _indeg(p)
    assert np.all(d[:8] == 0) and np.all((d[8:] >= 1) & (d[8:] <= 3))
    layer = np.arange(p.V) // 8
    for v in range(8, p.V):   # at least one predecessor from the previous layer
        assert np.any(layer[p.src[p.dst == v]] == layer[v] - 1)
    _check_dag_and_horizon(p, 1.5)


def test_random_layered():
    p = W.random_layered(1)
    assert p.V == 1000 and p.C == 4 and list(p.limit) == [8, 6, 4, 2]
    assert set(np.unique(p.lat)) <= {1, 2, 3, 4}
    frac = np.bincount(p.cls, minlength=4) / p.V
    np.testing.assert_allclose(frac, [0.4, 0.3, 0.2, 0.1], atol=0.05)
    d = _indeg(p)[25:]                       # non-source fan-in 1 + Poisson(1): mean 2, >= 1
    assert d.min() >= 1 and abs(d.mean() - 2.0) < 0.2
    _check_dag_and_horizon(p, 1.5)


def test_logic_network():
    p = W.logic_network(1)
    assert p.V == 10_000 and p.C == 2
    assert p.limit[0] == 64 and np.isinf(p.limit[1])
    assert np.all(p.lat == 1)
    d = _indeg(p)
    inner = d > 0
    # AND (class 0) takes exactly 2 inputs, INV (class 1) exactly 1; about 30 % INV
    assert np.all(d[inner & (p.cls == 0)] == 2) and np.all(d[inner & (p.cls == 1)] == 1)
    assert abs(np.mean(p.cls == 1) - 0.3) < 0.03
    assert _outdeg(p).max() <= 64
    assert p.cp == 120 and p.D == math.ceil(1.3 * 120) == 156
    assert 16_000 < p.E < 18_000
    _check_dag_and_horizon(p, None)


@pytest.mark.parametrize("factor", [1.0, 1.25, 1.5])
def test_modulo_loop(factor):
    p = W.modulo_loop(1, ii_factor=factor)
    assert p.V == 5000 and p.C == 6 and sorted(p.limit.tolist()) == [2, 4, 6, 8, 12, 16]
    assert set(np.unique(p.lat)) <= set(range(1, 7))
    assert 7000 < p.E < 9000 and p.NB == 200
    assert set(np.unique(p.bdist)) <= {1, 2, 3}
    assert p.D == 3 * p.II
    # II at least the resource bound max_c ceil(N_c / R_c)
    res_mii = max(math.ceil(np.sum(p.cls == c) / p.limit[c]) for c in range(p.C))
    assert p.II >= math.ceil(factor * res_mii) - 1
    # every back edge j -> i closes a cycle: i is an ancestor of j
    g = nx.DiGraph()
    g.add_edges_from(zip(p.src.tolist(), p.dst.tolist()))
    for j, i in zip(p.bsrc.tolist(), p.bdst.tolist()):
        assert nx.has_path(g, i, j)
    _check_dag_and_horizon(p, None)


def test_wide_layered():
    p = W.wide_layered(1)
    assert p.V == 50_000 and p.C == 8 and np.all(p.limit == 128)
    assert set(np.unique(p.lat)) <= set(range(1, 9))
    d = _indeg(p)[1000:]
    assert d.min() >= 2 and d.max() <= 4
    level = np.arange(p.V) // 1000
    gap = level[p.dst] - level[p.src]
    assert gap.min() >= 1 and gap.max() <= 3
    _check_dag_and_horizon(p, 1.4)
