"""Brute-force enumeration over every discrete schedule of a tiny DAG.

Independent of the oracle: bin masses come from scipy's ``ndtr`` (or, for the
other CDF families of App. D, scipy.stats' distributions) and the
discrete objectives are evaluated per schedule from the definitions of
Sec. 2.1 (Dep, Res, Mem, Rec) and App. B.1 (Com), then weighted by the
product of independent bin probabilities (Sec. 3.1-3.2).
"""
import itertools

import math

import numpy as np
from scipy import stats
from scipy.special import ndtr

# App. D scale matching, as the scipy `scale` of each family for sigma = 1:
# logistic s = sqrt(3)/pi and Laplace b = 1/sqrt(2) (unit variance), Cauchy
# gamma = sqrt(2 ln 2) (the normal's half width at half maximum)
FAMILY_CDF = {
    0: ndtr,
    1: lambda z: stats.logistic.cdf(z, scale=math.sqrt(3.0) / math.pi),
    2: lambda z: stats.laplace.cdf(z, scale=1.0 / math.sqrt(2.0)),
    3: lambda z: stats.cauchy.cdf(z, scale=math.sqrt(2.0 * math.log(2.0))),
}


def bin_probs(D, mu, sigma, family=0):
    """P{floor(X + 1/2) = d}, d = 0..D-1, open end bins, for X = mu + sigma Z with
    Z of the given family (0 normal, 1 logistic, 2 Laplace, 3 Cauchy)."""
    edges = (np.arange(D + 1) - 0.5 - mu) / sigma
    cdf = np.asarray(FAMILY_CDF[family](edges), dtype=np.float64)
    cdf[0] = 0.0
    cdf[-1] = 1.0
    return np.diff(cdf)


def discrete_metrics(p, s):
    """Per-schedule metrics over d in [0, D): dep count, com sum of (s_v - s_u)^+,
    usage counts per class, storage Mem(d), rec count."""
    D, V = p.D, p.V
    dep = sum(1 for u, v in zip(p.src, p.dst) if s[v] < s[u] + p.lat[u])
    com = sum(max(0, s[v] - s[u]) for u, v in zip(p.src, p.dst))
    use = np.zeros((p.C, D))
    for v in range(V):
        use[p.cls[v], s[v]] += p.demand[v]
    mem = np.zeros(D)
    for i in range(V):
        succ = [int(v) for u, v in zip(p.src, p.dst) if u == i]
        last = max(s[j] for j in succ) if succ else D
        for d in range(D):
            if s[i] <= d < last:
                mem[d] += p.bits[i]
    rec = 0
    for j, i, k in zip(p.bsrc, p.bdst, p.bdist):
        if s[i] + k * p.II < s[j] + p.lat[j]:
            rec += 1
    return dep, com, use, mem, rec


def expectations(p, mu, sigma, family=0):
    """Exact expectations by summing over all D^V schedules."""
    P = [bin_probs(p.D, mu[v], sigma[v], family) for v in range(p.V)]
    E = {"dep": 0.0, "com": 0.0, "use": np.zeros((p.C, p.D)), "mem": np.zeros(p.D), "rec": 0.0}
    for s in itertools.product(range(p.D), repeat=p.V):
        w = 1.0
        for v in range(p.V):
            w *= P[v][s[v]]
        if w == 0.0:
            continue
        dep, com, use, mem, rec = discrete_metrics(p, s)
        E["dep"] += w * dep
        E["com"] += w * com
        E["use"] += w * use
        E["mem"] += w * mem
        E["rec"] += w * rec
    return E


def fold(x, II):
    """App. B.3 fold: sum over k >= 0 of x[t + k II] for t in [0, II)."""
    if II <= 0:
        return x
    out = np.zeros(x.shape[:-1] + (II,))
    for d in range(x.shape[-1]):
        out[..., d % II] += x[..., d]
    return out
