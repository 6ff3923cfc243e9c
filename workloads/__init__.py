"""Seeded synthetic scheduling workloads for GauS (arXiv 2602.20427).

This module only builds inputs: a DAG with latencies, resource classes,
limits, demands, storage widths, optional back edges, a horizon D, an
initiation interval II and the initial (mu, sigma) of B restarts.  It holds
none of the method's arithmetic.  The one computation on the graph it performs
is a longest-path pass (``_longest_start``) that places the initial means near
each node's earliest start and sizes D from the critical path, as the
workload recipes prescribe; the library and the oracle compute their own
ASAP/ALAP independently.

The paper's benchmark suites (EPFL logic networks, GS-Schedule random
workloads) are not available here; the five generators below are synthetic
stand-ins with the graph shapes of those workloads (Sec. 4.1.2, App. C.2).
All randomness comes from ``numpy.random.default_rng(seed)``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# term bits, mirrored from the public header
DEP, COM, RES_OBJ, RES_VIOL, REG_OBJ, REC = 1, 2, 4, 8, 16, 32
DEP_CF = 64  # continuous dependency penalty (a variant, not the paper's Eq. dep)


@dataclass
class Problem:
    name: str
    V: int
    src: np.ndarray          # int32 (E,) producer
    dst: np.ndarray          # int32 (E,) consumer
    lat: np.ndarray          # int32 (V,)
    cls: np.ndarray          # int32 (V,)
    C: int
    limit: np.ndarray        # float64 (C,), inf = unlimited
    demand: np.ndarray       # int32 (V,)
    bits: np.ndarray         # int32 (V,)
    D: int
    II: int = 0
    bsrc: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int32))
    bdst: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int32))
    bdist: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int32))
    terms: int = DEP | COM | RES_OBJ
    B: int = 1
    lr: float = 1e-2
    iters: int = 1000

    @property
    def E(self) -> int:
        return int(self.src.size)

    @property
    def NB(self) -> int:
        return int(self.bsrc.size)


def _longest_start(V, src, dst, lat):
    """Earliest start of every node (nodes are generated in topological order)."""
    start = np.zeros(V, np.int64)
    order = np.argsort(dst, kind="stable")
    s_sorted, d_sorted = src[order], dst[order]
    ptr = np.searchsorted(d_sorted, np.arange(V + 1))
    for v in range(V):
        a, b = ptr[v], ptr[v + 1]
        if b > a:
            u = s_sorted[a:b]
            start[v] = np.max(start[u] + lat[u])
    return start


def _finish(name, V, src, dst, lat, cls, C, limit, rng, D=None, horizon=1.5, demand=None,
            bits=None, **kw):
    src = np.asarray(src, np.int32)
    dst = np.asarray(dst, np.int32)
    lat = np.asarray(lat, np.int32)
    start = _longest_start(V, src, dst, lat)
    cp = int(np.max(start + lat))
    if D is None:
        D = int(math.ceil(horizon * cp))
    p = Problem(name=name, V=V, src=src, dst=dst, lat=lat, cls=np.asarray(cls, np.int32),
                C=C, limit=np.asarray(limit, np.float64),
                demand=np.ones(V, np.int32) if demand is None else np.asarray(demand, np.int32),
                bits=np.ones(V, np.int32) if bits is None else np.asarray(bits, np.int32),
                D=D, **kw)
    p.start = start
    p.cp = cp
    return p


def init_state(p: Problem, B: int, seed: int, mu_jitter: str = "normal2", sigma0: float = 1.5):
    """Initial (mu, sigma) as float32 (V, B): mu around each node's earliest start."""
    rng = np.random.default_rng(seed + 7919)
    base = p.start.astype(np.float64)[:, None]
    if mu_jitter == "uniform01":
        mu = base + rng.uniform(0.0, 1.0, size=(p.V, B))
    else:
        mu = base + rng.normal(0.0, 2.0, size=(p.V, B))
    sigma = np.full((p.V, B), sigma0)
    return mu.astype(np.float32), sigma.astype(np.float32)


def tiny_layered(seed: int = 1) -> Problem:
    """|V| = 64 in 8 layers of 8; 1-3 distinct predecessors from earlier layers (at
    least one from the previous layer); 2 classes with limits 2 and 3; latencies
    uniform in {1, 2, 3}; D = ceil(1.5 * critical path); B = 1; lr 0.05."""
    rng = np.random.default_rng(seed)
    L, W = 8, 8
    V = L * W
    src, dst = [], []
    for layer in range(1, L):
        for k in range(W):
            v = layer * W + k
            n = int(rng.integers(1, 4))
            prev = layer * W - W + int(rng.integers(0, W))
            preds = {prev}
            pool = np.arange(0, layer * W)
            while len(preds) < n:
                preds.add(int(rng.choice(pool)))
            for u in sorted(preds):
                src.append(u)
                dst.append(v)
    lat = rng.integers(1, 4, size=V)
    cls = rng.integers(0, 2, size=V)
    return _finish("tiny_layered_v64", V, src, dst, lat, cls, 2, [2.0, 3.0], rng,
                   terms=DEP | COM | RES_OBJ | RES_VIOL, B=1, lr=0.05, iters=200)


def random_layered(seed: int = 1) -> Problem:
    """|V| = 1,000 in 40 layers of 25; fan-in 1 + Poisson(1) (at least one from the
    previous layer); 4 classes with probabilities .4/.3/.2/.1 and limits 8/6/4/2;
    latencies uniform in {1..4}; D = ceil(1.5 * critical path); B = 64."""
    rng = np.random.default_rng(seed)
    L, W = 40, 25
    V = L * W
    src, dst = [], []
    for layer in range(1, L):
        for k in range(W):
            v = layer * W + k
            n = min(1 + int(rng.poisson(1.0)), layer * W)
            preds = {layer * W - W + int(rng.integers(0, W))}
            while len(preds) < n:
                preds.add(int(rng.integers(0, layer * W)))
            for u in sorted(preds):
                src.append(u)
                dst.append(v)
    lat = rng.integers(1, 5, size=V)
    cls = rng.choice(4, size=V, p=[0.4, 0.3, 0.2, 0.1])
    return _finish("random_layered_v1000", V, src, dst, lat, cls, 4, [8.0, 6.0, 4.0, 2.0], rng,
                   terms=DEP | COM | RES_OBJ | RES_VIOL, B=64, iters=1000)


def logic_network(seed: int = 1, V: int = 10_000, depth: int = 120) -> Problem:
    """Logic-network-shaped DAG: |V| two-input AND and one-input INV nodes (30 % INV),
    depth levels of about V/depth nodes, level 0 sources.  Every non-source node
    has one predecessor in the previous level; an AND node's second predecessor
    lies 1 + Geometric(1/2) levels back.  Predecessors are drawn in proportion to
    a per-node Zipf(s = 1.5) fan-out weight, and no node feeds more than 64
    consumers.  Classes AND (limit 64) and INV (unlimited); all latencies 1;
    D = ceil(1.3 * depth); B = 64."""
    rng = np.random.default_rng(seed)
    per = V // depth
    sizes = np.full(depth, per)
    sizes[: V - per * depth] += 1
    offs = np.concatenate([[0], np.cumsum(sizes)])
    is_inv = rng.random(V) < 0.30
    weight = np.minimum(rng.zipf(1.5, size=V), 64).astype(np.float64)
    fanout = np.zeros(V, np.int64)
    src, dst = [], []

    def pick(level, exclude):
        lo, hi = offs[level], offs[level + 1]
        w = weight[lo:hi] * (fanout[lo:hi] < 64)
        for x in exclude:
            if lo <= x < hi:
                w[x - lo] = 0.0
        if w.sum() <= 0:
            w = (fanout[lo:hi] < 64).astype(np.float64)
            for x in exclude:
                if lo <= x < hi:
                    w[x - lo] = 0.0
        return lo + int(rng.choice(hi - lo, p=w / w.sum()))

    for level in range(1, depth):
        for v in range(offs[level], offs[level + 1]):
            u1 = pick(level - 1, ())
            preds = [u1]
            if not is_inv[v]:
                back = 1 + min(int(rng.geometric(0.5)) - 1, level - 1)
                preds.append(pick(level - back, (u1,)))
            for u in preds:
                fanout[u] += 1
                src.append(u)
                dst.append(v)
    cls = np.where(is_inv, 1, 0)
    lat = np.ones(V, np.int64)
    return _finish(f"logic_network_v{V}", V, src, dst, lat, cls, 2, [64.0, math.inf], rng,
                   D=int(math.ceil(1.3 * depth)), terms=DEP | COM | RES_OBJ | RES_VIOL,
                   B=64, iters=2000)


def _res_mii(p: Problem) -> int:
    mii = 1
    for c in range(p.C):
        if math.isfinite(p.limit[c]):
            n = int(p.demand[p.cls == c].sum())
            mii = max(mii, int(math.ceil(n / p.limit[c])))
    return mii


def _has_positive_cycle(V, src, dst, w) -> bool:
    """Bellman-Ford from a virtual source on edge weights w (longest-path sense)."""
    dist = np.zeros(V, np.int64)
    for _ in range(V):
        cand = dist[src] + w
        new = dist.copy()
        np.maximum.at(new, dst, cand)
        if np.array_equal(new, dist):
            return False
        dist = new
    return True


def modulo_loop(seed: int = 1, ii_factor: float = 1.0, V: int = 5000, levels: int = 50,
                n_back: int = 200) -> Problem:
    """Loop body for modulo scheduling: |V| nodes in `levels` levels, about 1.6 |V|
    intra-iteration edges (1-2 predecessors, one from the previous level), n_back
    loop-carried back edges j -> i (i an ancestor of j) with distance uniform in
    {1, 2, 3}; 6 classes with limits {2, 4, 6, 8, 12, 16}; latencies uniform in
    {1..6}.  II = ceil(ii_factor * MII) with MII = max(ResMII, RecMII); D = 3 II;
    B = 32."""
    rng = np.random.default_rng(seed)
    per = V // levels
    sizes = np.full(levels, per)
    sizes[: V - per * levels] += 1
    offs = np.concatenate([[0], np.cumsum(sizes)])
    src, dst = [], []
    for level in range(1, levels):
        for v in range(offs[level], offs[level + 1]):
            preds = {int(rng.integers(offs[level - 1], offs[level]))}
            if rng.random() < 0.63:
                preds.add(int(rng.integers(0, offs[level])))
            for u in sorted(preds):
                src.append(u)
                dst.append(v)
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    # back edges: pick j, walk up to 6 predecessor hops to an ancestor i
    pred_of = [[] for _ in range(V)]
    for u, v in zip(src, dst):
        pred_of[v].append(int(u))
    bsrc, bdst, bdist = [], [], []
    while len(bsrc) < n_back:
        j = int(rng.integers(offs[1], V))
        i = j
        for _ in range(int(rng.integers(1, 7))):
            if not pred_of[i]:
                break
            i = pred_of[i][int(rng.integers(0, len(pred_of[i])))]
        if i == j:
            continue
        bsrc.append(j)
        bdst.append(i)
        bdist.append(int(rng.integers(1, 4)))
    lat = rng.integers(1, 7, size=V)
    cls = rng.integers(0, 6, size=V)
    limit = [2.0, 4.0, 6.0, 8.0, 12.0, 16.0]
    p = _finish(f"modulo_loop_v{V}", V, src, dst, lat, cls, 6, limit, rng, D=1,
                bsrc=np.asarray(bsrc, np.int32), bdst=np.asarray(bdst, np.int32),
                bdist=np.asarray(bdist, np.int32),
                terms=DEP | RES_VIOL | REG_OBJ | REC, B=32, iters=2000)
    res_mii = _res_mii(p)
    # RecMII: least II without a positive cycle in the constraint graph
    fs = np.concatenate([src, np.asarray(bsrc)])
    fd = np.concatenate([dst, np.asarray(bdst)])
    lat64 = lat.astype(np.int64)

    def feasible(ii):
        w = np.concatenate([lat64[src], lat64[np.asarray(bsrc)] - np.asarray(bdist) * ii])
        return not _has_positive_cycle(V, fs, fd, w)

    lo, hi = 1, max(res_mii, 1)
    while not feasible(hi):
        hi *= 2
    while lo < hi:
        mid = (lo + hi) // 2
        if feasible(mid):
            hi = mid
        else:
            lo = mid + 1
    mii = max(res_mii, lo)
    p.II = int(math.ceil(ii_factor * mii))
    p.D = 3 * p.II
    p.mii = mii
    p.name = f"modulo_loop_v{V}_ii{p.II}"
    return p


def wide_layered(seed: int = 1, width: int = 1000, levels: int = 50) -> Problem:
    """Wide streaming-processor-shaped DAG: width * levels nodes; each node takes 2-4
    predecessors from the previous 1-3 levels; 8 classes with limit 128; latencies
    uniform in {1..8}; D = ceil(1.4 * critical path); B = 16; adds the
    register-lifetime objective (Formulation B)."""
    rng = np.random.default_rng(seed)
    V = width * levels
    src, dst = [], []
    for level in range(1, levels):
        for k in range(width):
            v = level * width + k
            n = int(rng.integers(2, 5))
            preds = {(level - 1) * width + int(rng.integers(0, width))}
            while len(preds) < n:
                back = int(rng.integers(1, min(3, level) + 1))
                preds.add((level - back) * width + int(rng.integers(0, width)))
            for u in sorted(preds):
                src.append(u)
                dst.append(v)
    lat = rng.integers(1, 9, size=V)
    cls = rng.integers(0, 8, size=V)
    return _finish(f"wide_layered_v{V}", V, src, dst, lat, cls, 8, [128.0] * 8, rng,
                   horizon=1.4, terms=DEP | RES_OBJ | RES_VIOL | REG_OBJ, B=16, iters=2000)


def random_small(seed: int, V: int, D: int, C: int = 2, max_lat: int = 2, p_edge: float = 0.3,
                 n_back: int = 0, II: int = 0) -> Problem:
    """Tiny random DAG for exhaustive checks: edge u -> v (u < v) with probability
    p_edge, latencies uniform in {0..max_lat}, demands and widths in {1, 2}."""
    rng = np.random.default_rng(seed)
    src, dst = [], []
    for v in range(1, V):
        for u in range(v):
            if rng.random() < p_edge:
                src.append(u)
                dst.append(v)
    lat = rng.integers(0, max_lat + 1, size=V)
    cls = rng.integers(0, C, size=V)
    limit = rng.integers(1, 3, size=C).astype(np.float64)
    bsrc, bdst, bdist = [], [], []
    for _ in range(n_back):
        j = int(rng.integers(1, V))
        i = int(rng.integers(0, j))
        bsrc.append(j)
        bdst.append(i)
        bdist.append(int(rng.integers(1, 3)))
    p = _finish(f"random_small_v{V}", V, src, dst, lat, cls, C, limit, rng, D=D,
                demand=rng.integers(1, 3, size=V), bits=rng.integers(1, 3, size=V),
                bsrc=np.asarray(bsrc, np.int32), bdst=np.asarray(bdst, np.int32),
                bdist=np.asarray(bdist, np.int32), II=II,
                terms=DEP | COM | RES_OBJ | RES_VIOL | REG_OBJ | (REC if II > 0 else 0))
    return p


CONFIGS = {
    "tiny": tiny_layered,
    "random": random_layered,
    "logic": logic_network,
    "modulo": modulo_loop,
    "wide": wide_layered,
}
