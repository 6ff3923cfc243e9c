"""Pins of the oracle's continuous dependency penalty (term DEP_CF).

DEP_CF is not the paper's binned Eq. dep: for the unrounded independent normals
X_u ~ N(mu_u, sigma_u^2), X_v ~ N(mu_v, sigma_v^2) it counts
P(X_u + Lat(u) > X_v) = Phi((mu_u + Lat(u) - mu_v) / sqrt(sigma_u^2 + sigma_v^2))
per edge, under the dependency multiplier.  Pinned against Monte Carlo sampling
of the continuous normals, quadrature of the defining integral with scipy, the
sigma -> 0 limit, the augmented-Lagrangian composition and central differences.
"""
import math

import numpy as np
import pytest
from scipy import integrate
from scipy.stats import norm

import oracle
import workloads as W


def _vdep(op, p, mu, sigma, terms=W.DEP_CF, **kw):
    _, T, _, _ = oracle.loss_grad(op, oracle.hparams(terms=terms, **kw), mu[:, None], sigma[:, None],
                                  np.zeros((1, 3)))
    return T[0, oracle.T_VDEP]


def test_equals_quadrature_of_the_definition():
    p = W.random_small(3, V=7, D=12, C=2, max_lat=3, p_edge=0.5)
    rng = np.random.default_rng(1)
    mu = rng.uniform(0, 11, p.V)
    sigma = rng.uniform(0.3, 3.0, p.V)
    ref = 0.0
    for u, v in zip(p.src, p.dst):
        # P(X_v < X_u + Lat(u)) = int f_u(x) F_v(x + Lat(u)) dx
        val, _ = integrate.quad(lambda x: norm.pdf(x, mu[u], sigma[u]) * norm.cdf(x + p.lat[u], mu[v], sigma[v]),
                                -np.inf, np.inf, epsabs=1e-13, epsrel=1e-12)
        ref += val
    assert _vdep(oracle.OracleProblem(p), p, mu, sigma) == pytest.approx(ref, abs=1e-9)


def test_monte_carlo_of_continuous_normals():
    p = W.random_small(4, V=8, D=10, C=2, max_lat=2, p_edge=0.4)
    rng = np.random.default_rng(2)
    mu, sigma = rng.uniform(0, 9, p.V), rng.uniform(0.5, 2.0, p.V)
    n = 400_000
    X = rng.normal(mu, sigma, size=(n, p.V))
    cnt = np.zeros(n)
    for u, v in zip(p.src, p.dst):
        cnt += X[:, u] + p.lat[u] > X[:, v]
    se = cnt.std() / math.sqrt(n)
    assert abs(cnt.mean() - _vdep(oracle.OracleProblem(p), p, mu, sigma)) < 4 * se


def test_small_sigma_limit_is_the_continuous_indicator():
    p = W.random_small(5, V=6, D=10, C=2, max_lat=2, p_edge=0.5)
    rng = np.random.default_rng(3)
    mu = rng.uniform(0, 9, p.V)
    # keep every margin |mu_u + Lat - mu_v| at least 0.05
    for u, v in zip(p.src, p.dst):
        if abs(mu[u] + p.lat[u] - mu[v]) < 0.05:
            mu[v] += 0.1
    sigma = np.full(p.V, 1e-4)
    want = sum(1.0 for u, v in zip(p.src, p.dst) if mu[u] + p.lat[u] > mu[v])
    assert _vdep(oracle.OracleProblem(p), p, mu, sigma) == pytest.approx(want, abs=1e-12)


def test_is_not_the_binned_term_but_agrees_where_rounding_cannot_matter():
    # a two-node chain far apart: both penalties vanish; at equal means they differ
    p = W.random_small(0, V=2, D=40, C=1, max_lat=1, p_edge=1.0)
    op = oracle.OracleProblem(p)
    far = np.array([5.0, 30.0]), np.array([1.0, 1.0])
    assert _vdep(op, p, *far) < 1e-12
    assert _vdep(op, p, *far, terms=W.DEP) < 1e-12
    near = np.array([10.0, 10.0]), np.array([1.0, 1.0])
    lat = p.lat[0]
    assert _vdep(op, p, *near) == pytest.approx(norm.cdf(lat / math.sqrt(2.0)), abs=1e-14)
    assert abs(_vdep(op, p, *near) - _vdep(op, p, *near, terms=W.DEP)) > 1e-3


def test_loss_composition_augmented_lagrangian():
    p = W.random_small(6, V=6, D=9, C=2, max_lat=2, p_edge=0.5)
    rng = np.random.default_rng(4)
    mu, sigma = rng.uniform(0, 8, p.V), rng.uniform(0.5, 2, p.V)
    op = oracle.OracleProblem(p)
    lam = np.array([[0.7, 0.0, 0.0]])
    hp = oracle.hparams(terms=W.DEP_CF, rho=0.3)
    loss, T, _, _ = oracle.loss_grad(op, hp, mu[:, None], sigma[:, None], lam)
    v = T[0, oracle.T_VDEP]
    assert loss[0] == pytest.approx(0.7 * v + 0.15 * v * v, rel=1e-14)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_gradient_matches_central_differences(seed):
    p = W.random_small(400 + seed, V=7, D=10, C=2, max_lat=2, p_edge=0.4)
    p.limit[:] = [0.6, 0.9]
    rng = np.random.default_rng(seed)
    mu = rng.uniform(0, p.D - 1, size=(p.V, 1))
    sigma = rng.uniform(0.5, 2.0, size=(p.V, 1))
    lam = rng.uniform(0.1, 1.0, size=(1, 3))
    op = oracle.OracleProblem(p)
    hp = oracle.hparams(tau=0.2, rho=0.5, alpha=0.7, w_res=1.3,
                        terms=W.DEP_CF | W.COM | W.RES_OBJ | W.RES_VIOL)
    U, _ = oracle.expected_hist(op, mu[:, 0], sigma[:, 0])
    assert np.min(np.abs(U - p.limit[:, None])) > 1e-4
    _, _, gm, gs = oracle.loss_grad(op, hp, mu, sigma, lam)
    h = 1e-6
    for v in range(p.V):
        for arr, g in ((mu, gm), (sigma, gs)):
            a = arr.copy(); a[v, 0] += h
            lp = oracle.loss_grad(op, hp, a if arr is mu else mu, a if arr is sigma else sigma, lam)[0][0]
            a[v, 0] -= 2 * h
            lm = oracle.loss_grad(op, hp, a if arr is mu else mu, a if arr is sigma else sigma, lam)[0][0]
            assert g[v, 0] == pytest.approx((lp - lm) / (2 * h), rel=1e-6, abs=1e-7)
