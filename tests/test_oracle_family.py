"""Pins of the oracle's CDF families (App. D) against facts fixed by mathematics.

The logistic, Laplace and Cauchy CDFs replace Phi in Eq. round with the scale
matched to sigma: logistic s = sigma sqrt(3)/pi and Laplace b = sigma/sqrt(2)
give the variance sigma^2; Cauchy gamma = sigma sqrt(2 ln 2) gives the normal's
full width at half maximum.  The pins: scipy's distributions, unit mass, unit
variance and the half maximum by quadrature, the density as the CDF's
derivative, exhaustive enumeration of the expectations and central differences
of the full loss.
"""
import math

import numpy as np
import pytest
from scipy import integrate

import oracle
import workloads as W
from tests import _enumerate as EN

FAMILIES = (oracle.LOGISTIC, oracle.LAPLACE, oracle.CAUCHY)
ALL = (oracle.GAUSSIAN,) + FAMILIES


@pytest.mark.parametrize("fam", ALL)
def test_cdf_matches_scipy_and_is_symmetric(fam):
    for z in np.linspace(-12, 12, 49):
        F = oracle.F(fam, z)
        assert F == pytest.approx(float(EN.FAMILY_CDF[fam](z)), rel=1e-12, abs=1e-300)
        assert F + oracle.F(fam, -z) == pytest.approx(1.0, abs=1e-15)
    assert oracle.F(fam, 0.0) == 0.5


@pytest.mark.parametrize("fam", ALL)
def test_density_is_the_derivative_of_the_cdf(fam):
    h = 1e-5
    for z in np.linspace(-9, 9, 37):
        if fam == oracle.LAPLACE and abs(z) < 2 * h:
            continue  # the Laplace density has a kink at the centre
        x = -abs(z)  # the lower tail keeps the difference quotient accurate
        fd = (oracle.F(fam, x + h) - oracle.F(fam, x - h)) / (2 * h)
        assert oracle.f(fam, z) == pytest.approx(fd, rel=1e-7, abs=1e-13)
        assert oracle.f(fam, z) == oracle.f(fam, -z)


@pytest.mark.parametrize("fam", ALL)
def test_unit_mass(fam):
    m, _ = integrate.quad(lambda z: oracle.f(fam, z), -np.inf, np.inf, limit=400)
    assert m == pytest.approx(1.0, abs=1e-9)


@pytest.mark.parametrize("fam", (oracle.GAUSSIAN, oracle.LOGISTIC, oracle.LAPLACE))
def test_variance_matching(fam):
    # App. D: logistic and Laplace scales chosen for the variance sigma^2 (sigma = 1 here)
    var, _ = integrate.quad(lambda z: z * z * oracle.f(fam, z), -np.inf, np.inf, limit=400)
    assert var == pytest.approx(1.0, rel=1e-9)


def test_cauchy_half_width_matching():
    # App. D: the Cauchy scale matches the normal's FWHM 2 sqrt(2 ln 2) sigma
    hw = math.sqrt(2.0 * math.log(2.0))
    for fam in (oracle.GAUSSIAN, oracle.CAUCHY):
        assert oracle.f(fam, hw) / oracle.f(fam, 0.0) == pytest.approx(0.5, rel=1e-14)
    # ... and the Cauchy has no finite variance: the truncated second moment keeps growing
    m = [integrate.quad(lambda z: z * z * oracle.f(oracle.CAUCHY, z), -L, L, limit=400)[0]
         for L in (1e2, 1e3)]
    assert m[1] > 5 * m[0]


@pytest.mark.parametrize("fam", ALL)
@pytest.mark.parametrize("D", [1, 2, 7, 64])
def test_bin_masses_sum_to_one_and_match_library(fam, D):
    rng = np.random.default_rng(10 * D + fam)
    for _ in range(30):
        mu = rng.uniform(-20, D + 20)
        sigma = 10 ** rng.uniform(-2, 1.5)
        P = oracle.bin_masses(D, mu, sigma, fam)
        assert np.all(P >= -1e-15)
        assert abs(P.sum() - 1.0) < 1e-12
        np.testing.assert_allclose(P, EN.bin_probs(D, mu, sigma, fam), atol=1e-13)


def test_heavier_tails_than_the_normal():
    # at equal sigma, the far tail mass orders Gaussian < logistic < Laplace < Cauchy
    q = [oracle.F(fam, -6.0) for fam in ALL]
    assert q[0] < q[1] < q[2] < q[3]


@pytest.mark.parametrize("fam", FAMILIES)
@pytest.mark.parametrize("case", [0, 3, 6])
def test_expectations_equal_exhaustive_enumeration(fam, case):
    if case < 6:
        p = W.random_small(case, V=3 + case % 3, D=4 + case % 2, C=2, max_lat=2, p_edge=0.5)
    else:
        p = W.random_small(100, V=4, D=6, C=2, max_lat=2, p_edge=0.5, n_back=2, II=3)
    rng = np.random.default_rng(2000 + case + 10 * fam)
    mu = rng.uniform(-0.5, p.D - 0.5, size=p.V)
    sigma = rng.uniform(0.4, 2.0, size=p.V)
    op = oracle.OracleProblem(p)
    terms = W.DEP | W.COM | W.RES_OBJ | W.REG_OBJ | (W.REC if p.II else 0)
    hp = oracle.hparams(tau=0.3, terms=terms, family=fam)
    _, T, _, _ = oracle.loss_grad(op, hp, mu[:, None], sigma[:, None], np.zeros((1, 3)))
    E = EN.expectations(p, mu, sigma, fam)
    assert T[0, oracle.T_VDEP] == pytest.approx(E["dep"], abs=1e-12)
    assert T[0, oracle.T_COM] == pytest.approx(E["com"], abs=1e-12)
    if p.II:
        assert T[0, oracle.T_VREC] == pytest.approx(E["rec"], abs=1e-12)
    U, R = oracle.expected_hist(op, mu, sigma, fam)
    np.testing.assert_allclose(U, EN.fold(E["use"], p.II), atol=1e-12)
    np.testing.assert_allclose(R, EN.fold(E["mem"], p.II), atol=1e-12)


@pytest.mark.parametrize("fam", FAMILIES)
@pytest.mark.parametrize("II", [0, 4])
def test_gradient_matches_central_differences(fam, II):
    p = W.random_small(300 + II + fam, V=7, D=10, C=2, max_lat=2, p_edge=0.4,
                       n_back=3 if II else 0, II=II)
    p.limit[:] = [0.6, 0.9]
    rng = np.random.default_rng(fam)
    mu = rng.uniform(0, p.D - 1, size=(p.V, 1))
    sigma = rng.uniform(0.5, 2.0, size=(p.V, 1))
    lam = rng.uniform(0.1, 1.0, size=(1, 3))
    op = oracle.OracleProblem(p)
    terms = W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL | W.REG_OBJ | (W.REC if II else 0)
    hp = oracle.hparams(tau=0.2, rho=0.5, alpha=0.7, w_res=1.3, w_mem=0.8, terms=terms, family=fam)
    U, _ = oracle.expected_hist(op, mu[:, 0], sigma[:, 0], fam)
    assert np.min(np.abs(U - p.limit[:, None])) > 1e-4   # stay off the ReLU kinks
    _, _, gm, gs = oracle.loss_grad(op, hp, mu, sigma, lam)
    h = 1e-6
    for v in range(p.V):
        for arr, g in ((mu, gm), (sigma, gs)):
            a = arr.copy(); a[v, 0] += h
            lp = oracle.loss_grad(op, hp, a if arr is mu else mu, a if arr is sigma else sigma, lam)[0][0]
            a[v, 0] -= 2 * h
            lm = oracle.loss_grad(op, hp, a if arr is mu else mu, a if arr is sigma else sigma, lam)[0][0]
            fd = (lp - lm) / (2 * h)
            assert g[v, 0] == pytest.approx(fd, rel=1e-6, abs=1e-7)


def test_family_changes_the_loss():
    # a planted mistake that ignored the family would leave every loss equal
    p = W.random_small(5, V=6, D=9, C=2, max_lat=2, p_edge=0.5)
    rng = np.random.default_rng(9)
    mu = rng.uniform(0, 8, size=(p.V, 1))
    sigma = rng.uniform(0.5, 2.0, size=(p.V, 1))
    op = oracle.OracleProblem(p)
    losses = [oracle.loss_grad(op, oracle.hparams(terms=W.DEP | W.COM, family=fam), mu, sigma,
                               np.zeros((1, 3)))[0][0] for fam in ALL]
    assert len(set(np.round(losses, 12))) == 4
