"""Exhaustive optimal schedules of tiny DAGs against the oracle.

Every schedule in [0, D)^V is enumerated (numpy); legality and the
Formulation A objective L_Res + alpha L_Com (Sec. 4.1.1) are evaluated from the
discrete definitions.  The oracle's verifier must agree on every schedule's
legality and objective, and a short GauS run driven by the oracle (Alg. GauS:
loss, Adam, lambda update, round, Alg. 1) must end on a legal schedule no
better than the exhaustive optimum.  The optimality gap is printed, not gated.
"""
import itertools

import numpy as np
import pytest

import oracle
import workloads as W


def all_schedules(V, D):
    return np.array(list(itertools.product(range(D), repeat=V)), dtype=np.int64)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_exhaustive_optimum_formulation_a(seed):
    p = W.random_small(300 + seed, V=6, D=5, C=2, max_lat=1, p_edge=0.35)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    assert rc == 0
    S = all_schedules(p.V, p.D)
    legal = np.ones(len(S), bool)
    for u, v in zip(p.src, p.dst):
        legal &= S[:, v] >= S[:, u] + p.lat[u]
    legal &= np.all(S + p.lat[None, :] <= p.D, axis=1)
    com = np.zeros(len(S), np.int64)
    for u, v in zip(p.src, p.dst):
        com += S[:, v] - S[:, u]
    lres = np.zeros(len(S), np.int64)
    for c in range(p.C):
        cnt = np.zeros((len(S), p.D), np.int64)
        for v in np.nonzero(p.cls == c)[0]:
            cnt[np.arange(len(S)), S[:, v]] += p.demand[v]
        lres += cnt.max(axis=1)
    obj = lres + com
    rng = np.random.default_rng(seed)
    for idx in rng.choice(len(S), size=200, replace=False):
        rep = oracle.verify(op, S[idx].astype(np.int32))
        assert rep["feasible"] == int(legal[idx])
        assert rep["L_res"] + rep["L_com"] == obj[idx]
    best = obj[legal].min()

    # GauS (Alg. GauS) with the oracle: init mu = (ASAP + ALAP)/2, sigma = kappa (ALAP - ASAP)
    mu = ((asap + alap) / 2.0)[:, None]
    sg = np.maximum((alap - asap) / 6.0, 0.05)[:, None]
    m1, v1, m2, v2 = (np.zeros((p.V, 1)) for _ in range(4))
    lam = np.full((1, 3), 1e-6)
    hp = oracle.hparams(tau=1e-2, rho=1e-4, alpha=1.0, terms=W.DEP | W.COM | W.RES_OBJ)
    found = None
    for step in range(1, 301):
        loss, T, gm, gs = oracle.loss_grad(op, hp, mu, sg, lam)
        for th, g, m, v in ((mu, gm, m1, v1), (sg, gs, m2, v2)):
            oracle.adam(th.reshape(-1), np.ascontiguousarray(g.reshape(-1)), m.reshape(-1),
                        v.reshape(-1), step, 0.05)
        np.maximum(sg, 0.05, out=sg)
        lam[0, 0] += 1e-4 * T[0, oracle.T_VDEP]
        s = oracle.legalize_regular(op, order, asap, alap, oracle.round_half_up(mu[:, 0]))
        rep = oracle.verify(op, s)
        assert rep["feasible"] == 1
        val = rep["L_res"] + rep["L_com"]
        found = val if found is None else min(found, val)
    assert found >= best
    print(f"seed {seed}: exhaustive optimum {best}, GauS-oracle best {found}")
