"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: library
routines (scipy, networkx, torch.optim.Adam), exhaustive enumeration over every
discrete schedule, Monte Carlo sampling of rounded Gaussians, finite
differences, closed forms and degenerate cases.
"""
import math

import networkx as nx
import numpy as np
import pytest
from scipy.special import logsumexp, ndtr

import oracle
import workloads as W
from tests import _enumerate as EN

ALL_TERMS = W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL | W.REG_OBJ


# ---------------------------------------------------------------- Phi, Eq. round
def test_phi_matches_library_and_symmetry():
    for z in np.linspace(-8, 8, 33):
        assert oracle.Phi(z) == pytest.approx(ndtr(z), rel=1e-13, abs=1e-300)
        assert oracle.Phi(z) + oracle.Phi(-z) == pytest.approx(1.0, abs=1e-15)
        assert oracle.phi(z) == pytest.approx(math.exp(-z * z / 2) / math.sqrt(2 * math.pi), rel=1e-14)
    assert oracle.Phi(0.0) == 0.5


def test_three_sigma_mass_kappa_one_sixth():
    # App. D: kappa = 1/6 puts +-3 sigma at the [ASAP, ALAP] ends, ~99.7 % of the mass
    m = oracle.Phi(3.0) - oracle.Phi(-3.0)
    assert m == pytest.approx(0.9973002039367398, abs=1e-13)


@pytest.mark.parametrize("D", [1, 2, 5, 37, 200])
def test_bin_masses_sum_to_one_and_match_library(D):
    rng = np.random.default_rng(D)
    for _ in range(50):
        mu = rng.uniform(-30, D + 30)
        sigma = 10 ** rng.uniform(-3, 1.5)
        P = oracle.bin_masses(D, mu, sigma)
        assert np.all(P >= -1e-15)
        assert abs(P.sum() - 1.0) < 1e-12          # open end bins (Sec. 3.2 footnote)
        np.testing.assert_allclose(P, EN.bin_probs(D, mu, sigma), atol=1e-14)


def test_round_half_up():
    mu = np.array([-1.5, -0.5, -0.49999997, 0.0, 0.49999997, 0.5, 1.5, 2.4999998, 7.5],
                  dtype=np.float32).astype(np.float64)
    np.testing.assert_array_equal(oracle.round_half_up(mu), [-1, 0, 0, 0, 0, 1, 2, 2, 8])


# ---------------------------------------------------------------- expectations
def _tiny_cases():
    cases = []
    for seed in range(6):
        V = 3 + seed % 3
        D = 4 + seed % 2
        cases.append(W.random_small(seed, V=V, D=D, C=2, max_lat=2, p_edge=0.5))
    # modulo cases with back edges
    for seed in range(3):
        cases.append(W.random_small(100 + seed, V=4, D=6, C=2, max_lat=2, p_edge=0.5,
                                    n_back=2, II=3))
    return cases


@pytest.mark.parametrize("case", range(9))
def test_expectations_equal_exhaustive_enumeration(case):
    p = _tiny_cases()[case]
    rng = np.random.default_rng(1000 + case)
    mu = rng.uniform(-0.5, p.D - 0.5, size=p.V)
    sigma = rng.uniform(0.4, 2.0, size=p.V)
    op = oracle.OracleProblem(p)
    terms = W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL | W.REG_OBJ | (W.REC if p.II else 0)
    hp = oracle.hparams(tau=0.3, terms=terms)
    loss, T, _, _ = oracle.loss_grad(op, hp, mu[:, None], sigma[:, None], np.zeros((1, 3)))
    E = EN.expectations(p, mu, sigma)
    assert T[0, oracle.T_VDEP] == pytest.approx(E["dep"], abs=1e-12)
    assert T[0, oracle.T_COM] == pytest.approx(E["com"], abs=1e-12)
    if p.II:
        assert T[0, oracle.T_VREC] == pytest.approx(E["rec"], abs=1e-12)
    U, R = oracle.expected_hist(op, mu, sigma)
    np.testing.assert_allclose(U, EN.fold(E["use"], p.II), atol=1e-12)
    np.testing.assert_allclose(R, EN.fold(E["mem"], p.II), atol=1e-12)
    # LogSumExp objective (Eq. max) and ReLU violation (Eq. relu) of those expectations
    Uf = EN.fold(E["use"], p.II)
    lse = sum(0.3 * logsumexp(Uf[c] / 0.3) for c in range(p.C))
    assert T[0, oracle.T_RES] == pytest.approx(lse, abs=1e-10)
    relu = sum(np.maximum(Uf[c] - p.limit[c], 0).sum() for c in range(p.C))
    assert T[0, oracle.T_VRES] == pytest.approx(relu, abs=1e-12)
    assert T[0, oracle.T_REG] == pytest.approx(0.3 * logsumexp(EN.fold(E["mem"], p.II) / 0.3),
                                               abs=1e-10)


def test_eq_dep_is_the_zero_latency_case():
    # Eq. dep counts d_j < d_i; with Lat = 0 the latency reading must coincide
    p = W.random_small(7, V=5, D=6, p_edge=0.6)
    p.lat[:] = 0
    rng = np.random.default_rng(3)
    mu, sigma = rng.uniform(0, 5, p.V), rng.uniform(0.5, 2, p.V)
    P = [EN.bin_probs(p.D, mu[v], sigma[v]) for v in range(p.V)]
    ref = 0.0
    for i, j in zip(p.src, p.dst):
        for di in range(1, p.D):
            for dj in range(0, di):
                ref += P[i][di] * P[j][dj]
    op = oracle.OracleProblem(p)
    _, T, _, _ = oracle.loss_grad(op, oracle.hparams(terms=W.DEP), mu[:, None], sigma[:, None],
                                  np.zeros((1, 3)))
    assert T[0, oracle.T_VDEP] == pytest.approx(ref, abs=1e-13)


def test_monte_carlo_of_rounded_gaussians():
    p = W.random_small(11, V=6, D=8, C=2, p_edge=0.4)
    rng = np.random.default_rng(5)
    mu, sigma = rng.uniform(0, 7, p.V), rng.uniform(0.5, 1.5, p.V)
    op = oracle.OracleProblem(p)
    _, T, _, _ = oracle.loss_grad(op, oracle.hparams(terms=W.DEP | W.COM), mu[:, None],
                                  sigma[:, None], np.zeros((1, 3)))
    U, R = oracle.expected_hist(op, mu, sigma)
    n = 200_000
    X = rng.normal(mu, sigma, size=(n, p.V))
    S = np.clip(np.floor(X + 0.5), 0, p.D - 1).astype(np.int64)   # open end bins
    dep = np.zeros(n)
    com = np.zeros(n)
    for u, v in zip(p.src, p.dst):
        dep += S[:, v] < S[:, u] + p.lat[u]
        com += np.maximum(S[:, v] - S[:, u], 0)
    for val, est in ((T[0, oracle.T_VDEP], dep), (T[0, oracle.T_COM], com)):
        se = est.std() / math.sqrt(n)
        assert abs(est.mean() - val) < 4 * se + 1e-9
    # usage of class 0 at every step
    for d in range(p.D):
        cnt = ((S == d) * (p.cls == 0) * p.demand).sum(axis=1)
        se = cnt.std() / math.sqrt(n)
        assert abs(cnt.mean() - U[0, d]) < 4 * se + 1e-9


# ---------------------------------------------------------------- gradient
@pytest.mark.parametrize("seed,II", [(0, 0), (1, 0), (2, 0), (3, 4), (4, 5)])
def test_gradient_matches_central_differences(seed, II):
    p = W.random_small(200 + seed, V=7, D=10, C=2, max_lat=2, p_edge=0.4,
                       n_back=3 if II else 0, II=II)
    p.limit[:] = [0.6, 0.9]
    rng = np.random.default_rng(seed)
    mu = rng.uniform(0, p.D - 1, size=(p.V, 1))
    sigma = rng.uniform(0.5, 2.0, size=(p.V, 1))
    lam = rng.uniform(0.1, 1.0, size=(1, 3))
    op = oracle.OracleProblem(p)
    terms = ALL_TERMS | (W.REC if II else 0)
    hp = oracle.hparams(tau=0.2, rho=0.5, alpha=0.7, w_res=1.3, w_mem=0.8, terms=terms)
    U, _ = oracle.expected_hist(op, mu[:, 0], sigma[:, 0])
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


def test_loss_composition_augmented_lagrangian():
    # Sec. 3.3: L = objectives + sum_k lambda_k V_k + rho/2 V_k^2
    p = W.random_small(31, V=5, D=7, p_edge=0.5)
    rng = np.random.default_rng(2)
    mu, sg = rng.uniform(0, 6, (p.V, 1)), rng.uniform(0.5, 2, (p.V, 1))
    lam = np.array([[0.3, 0.7, 0.0]])
    hp = oracle.hparams(tau=0.1, rho=0.25, alpha=0.5, w_res=2.0, w_mem=1.5, terms=ALL_TERMS)
    loss, T, _, _ = oracle.loss_grad(oracle.OracleProblem(p), hp, mu, sg, lam)
    t = T[0]
    ref = 2.0 * t[0] + 0.5 * t[1] + 1.5 * t[2] + 0.3 * t[3] + 0.125 * t[3] ** 2 \
        + 0.7 * t[4] + 0.125 * t[4] ** 2
    assert loss[0] == pytest.approx(ref, rel=1e-14)


# ---------------------------------------------------------------- degenerate case
def test_one_hot_limit_ties_expectations_to_verifier():
    # sigma -> 0 with integer mu makes every P one-hot: each expected term equals
    # the verifier's discrete value, and LSE_tau -> max as tau -> 0 (Eq. max)
    p = W.logic_network(3, V=300, depth=12)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    rng = np.random.default_rng(4)
    s = np.clip(asap + rng.integers(0, 3, p.V), 0, p.D - 1).astype(np.int32)
    mu = s.astype(np.float64)[:, None]
    sigma = np.full((p.V, 1), 1e-4)
    hp = oracle.hparams(tau=1e-3, terms=W.DEP | W.COM | W.RES_OBJ | W.REG_OBJ)
    _, T, _, _ = oracle.loss_grad(op, hp, mu, sigma, np.zeros((1, 3)))
    rep = oracle.verify(op, s)
    assert T[0, oracle.T_VDEP] == pytest.approx(rep["n_dep_viol"], abs=1e-9)
    com_pos = sum(max(0, s[v] - s[u]) for u, v in zip(p.src, p.dst))
    assert T[0, oracle.T_COM] == pytest.approx(com_pos, abs=1e-9)
    if rep["n_dep_viol"] == 0:
        assert com_pos == rep["L_com"]
    tau, D = 1e-3, p.D
    assert rep["L_res"] <= T[0, oracle.T_RES] + 1e-9
    assert T[0, oracle.T_RES] <= rep["L_res"] + p.C * tau * math.log(D) + 1e-9
    assert rep["L_mem"] <= T[0, oracle.T_REG] + 1e-9 <= rep["L_mem"] + tau * math.log(D) + 2e-9
    U, R = oracle.expected_hist(op, mu[:, 0], sigma[:, 0])
    cnt = np.zeros((p.C, p.D))
    for v in range(p.V):
        cnt[p.cls[v], s[v]] += p.demand[v]
    np.testing.assert_allclose(U, cnt, atol=1e-9)


# ---------------------------------------------------------------- ASAP / ALAP
def _nx_longest(p, D):
    G = nx.DiGraph()
    G.add_nodes_from(range(p.V))
    G.add_node("S")
    G.add_node("T")
    for v in range(p.V):
        G.add_edge("S", v, w=0)
        G.add_edge(v, "T", w=-int(p.lat[v]))
    for u, v in zip(p.src, p.dst):
        G.add_edge(int(u), int(v), w=-int(p.lat[u]))
    asap = nx.single_source_bellman_ford_path_length(G, "S", weight="w")
    R = G.reverse()
    tail = nx.single_source_bellman_ford_path_length(R, "T", weight="w")
    return (np.array([-asap[v] for v in range(p.V)]),
            np.array([D + tail[v] for v in range(p.V)]))


@pytest.mark.parametrize("gen", ["tiny", "random", "modulo_small"])
def test_asap_alap_against_networkx(gen):
    if gen == "tiny":
        p = W.tiny_layered(2)
    elif gen == "random":
        p = W.random_layered(2)
    else:
        p = W.random_small(9, V=30, D=40, p_edge=0.2, max_lat=3)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    assert rc == 0
    ra, rl = _nx_longest(p, p.D)
    np.testing.assert_array_equal(asap, ra)
    np.testing.assert_array_equal(alap, rl)
    assert cp == int(np.max(ra + p.lat))
    # the order is topological
    pos = np.empty(p.V, int)
    pos[order] = np.arange(p.V)
    assert np.all(pos[p.src] < pos[p.dst])


def test_asap_alap_errors():
    p = W.random_small(1, V=4, D=5, p_edge=1.0)
    p2 = W.Problem("cyc", 3, np.array([0, 1, 2], np.int32), np.array([1, 2, 0], np.int32),
                   np.ones(3, np.int32), np.zeros(3, np.int32), 1, np.array([1.0]),
                   np.ones(3, np.int32), np.ones(3, np.int32), D=10)
    assert oracle.asap_alap(oracle.OracleProblem(p2))[0] == 1
    p.D = 1
    p.lat[:] = 2
    assert oracle.asap_alap(oracle.OracleProblem(p))[0] == 2


# ---------------------------------------------------------------- Alg. 1
def _random_topo_order(p, rng):
    indeg = np.bincount(p.dst, minlength=p.V)
    ready = [v for v in range(p.V) if indeg[v] == 0]
    out = []
    succ = [[] for _ in range(p.V)]
    for u, v in zip(p.src, p.dst):
        succ[u].append(int(v))
    while ready:
        v = ready.pop(int(rng.integers(0, len(ready))))
        out.append(v)
        for w in succ[v]:
            indeg[w] -= 1
            if indeg[w] == 0:
                ready.append(w)
    return np.array(out, np.int32)


def test_alg1_legal_bounded_idempotent_order_free():
    p = W.random_layered(4)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    rng = np.random.default_rng(0)
    for trial in range(5):
        s0 = rng.integers(-5, p.D + 5, size=p.V).astype(np.int32)
        s1 = oracle.legalize_regular(op, order, asap, alap, s0)
        rep = oracle.verify(op, s1)
        assert rep["n_dep_viol"] == 0 and rep["n_lat_viol"] == 0
        assert np.all(s1 >= asap) and np.all(s1 <= alap)
        np.testing.assert_array_equal(oracle.legalize_regular(op, order, asap, alap, s1), s1)
        other = _random_topo_order(p, rng)
        np.testing.assert_array_equal(oracle.legalize_regular(op, other, asap, alap, s0), s1)


def test_alg1_is_least_legal_schedule_above_clamp():
    import itertools
    p = W.random_small(21, V=5, D=7, p_edge=0.5, max_lat=2)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    assert rc == 0
    rng = np.random.default_rng(1)
    for _ in range(10):
        s0 = rng.integers(0, p.D, size=p.V).astype(np.int32)
        c = np.clip(s0, asap, alap)
        best = None
        for s in itertools.product(*[range(c[v], p.D) for v in range(p.V)]):
            s = np.array(s)
            if all(s[v] >= s[u] + p.lat[u] for u, v in zip(p.src, p.dst)):
                best = s if best is None else np.minimum(best, s)
        # the componentwise minimum of the legal set above c is itself legal and least
        np.testing.assert_array_equal(oracle.legalize_regular(op, order, asap, alap, s0), best)


# ---------------------------------------------------------------- Alg. 2
def test_alg2_least_fixed_point_equals_bellman_ford():
    p = W.modulo_loop(3, V=400, levels=20, n_back=20)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    rng = np.random.default_rng(7)
    s0 = rng.integers(-3, p.D, size=p.V).astype(np.int32)
    s1, rc2 = oracle.legalize_modulo(op, order, s0)
    assert rc2 == 0
    # longest path from a source with edge S -> v of weight max(s0_v, 0)
    G = nx.DiGraph()
    for v in range(p.V):
        G.add_edge("S", v, w=-max(int(s0[v]), 0))
    for u, v in zip(p.src, p.dst):
        G.add_edge(int(u), int(v), w=-int(p.lat[u]))
    for j, i, k in zip(p.bsrc, p.bdst, p.bdist):
        G.add_edge(int(j), int(i), w=-(int(p.lat[j]) - int(k) * p.II))
    dist = nx.single_source_bellman_ford_path_length(G, "S", weight="w")
    np.testing.assert_array_equal(s1, [-dist[v] for v in range(p.V)])
    rep = oracle.verify(op, s1)
    assert rep["n_dep_viol"] == 0 and rep["n_rec_viol"] == 0


def test_alg2_reports_positive_cycle():
    p = W.random_small(5, V=4, D=8, p_edge=1.0, max_lat=1)
    p.lat[:] = 1
    p.bsrc = np.array([3], np.int32)
    p.bdst = np.array([0], np.int32)
    p.bdist = np.array([1], np.int32)
    p.II = 1      # the path 0 -> ... -> 3 needs >= 3 steps, so II = 1 is infeasible
    op = oracle.OracleProblem(p)
    rc, order, *_ = oracle.asap_alap(op)
    _, rc2 = oracle.legalize_modulo(op, order, np.zeros(p.V, np.int32))
    assert rc2 == 1


# ---------------------------------------------------------------- Adam
def test_adam_matches_torch_and_first_step_closed_form():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    n = 17
    th0 = rng.normal(size=n)
    grads = [rng.normal(size=n) * 10 ** rng.uniform(-3, 1) for _ in range(6)]
    th, m, v = th0.copy(), np.zeros(n), np.zeros(n)
    t = torch.tensor(th0.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.Adam([t], lr=0.05, betas=(0.9, 0.999), eps=1e-8)
    for step, g in enumerate(grads, 1):
        oracle.adam(th, np.ascontiguousarray(g), m, v, step, 0.05)
        t.grad = torch.tensor(g)
        opt.step()
        np.testing.assert_allclose(th, t.detach().numpy(), rtol=1e-14, atol=1e-15)
        if step == 1:
            np.testing.assert_allclose(th, th0 - 0.05 * g / (np.abs(g) + 1e-8), rtol=1e-13)


def test_upper_tail_bin_masses_keep_relative_accuracy():
    # far above the mean the masses come from the upper tails (1 - Phi loses them to
    # cancellation): compare with scipy's survival function
    from scipy.stats import norm
    P = oracle.bin_masses(14, 0.0, 1.0)
    for d in range(7, 13):
        ref = norm.sf(d - 0.5) - norm.sf(d + 0.5)
        assert P[d] == pytest.approx(ref, rel=1e-12)
    assert P[13] == pytest.approx(norm.sf(12.5), rel=1e-12)
    # and below the mean from the lower tails, by symmetry
    Q = oracle.bin_masses(14, 13.0, 1.0)
    for d in range(1, 7):
        assert Q[d] == pytest.approx(norm.cdf(d + 0.5 - 13.0) - norm.cdf(d - 0.5 - 13.0), rel=1e-12)


@pytest.mark.parametrize("tau", [0.01, 0.3, 2.0])
def test_lse_bounds(tau):
    # Eq. max: max_d x_d <= LSE_tau(x) <= max_d x_d + tau ln(#bins), per class and for storage
    p = W.random_small(41, V=9, D=12, C=3, max_lat=2, p_edge=0.3)
    rng = np.random.default_rng(int(tau * 100))
    mu, sigma = rng.uniform(0, 11, p.V), rng.uniform(0.3, 2.0, p.V)
    op = oracle.OracleProblem(p)
    _, T, _, _ = oracle.loss_grad(op, oracle.hparams(tau=tau, terms=W.RES_OBJ | W.REG_OBJ), mu[:, None],
                                  sigma[:, None], np.zeros((1, 3)))
    U, R = oracle.expected_hist(op, mu, sigma)
    lo = U.max(axis=1).sum()
    assert lo - 1e-12 <= T[0, oracle.T_RES] <= lo + p.C * tau * math.log(p.D) + 1e-12
    assert R.max() - 1e-12 <= T[0, oracle.T_REG] <= R.max() + tau * math.log(p.D) + 1e-12
