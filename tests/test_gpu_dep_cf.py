"""GPU path with the continuous dependency penalty (term DEP_CF; a variant, not the
paper's binned Eq. dep) against the fp64 oracle, through the C ABI, with the
tolerances of the normal's parity tests."""
import numpy as np
import pytest

import oracle
import workloads as W

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from tests.test_gpu_parity import _lam, check_loss_grad  # noqa: E402


@pytest.fixture(scope="module")
def g():
    import paper_2602_20427_gb300 as g
    g.build()
    g.lib()
    return g


def _cf(terms):
    return (terms & ~W.DEP) | W.DEP_CF


@pytest.mark.parametrize("B", [1, 5])
def test_tiny_layered(g, B):
    p = W.tiny_layered(1)
    mu, sg = W.init_state(p, B, 1, mu_jitter="uniform01", sigma0=1.0)
    hp = g.default_hparams(terms=_cf(p.terms), tau=0.05, rho=0.01)
    check_loss_grad(p, g, B, mu, sg, _lam(B, np.random.default_rng(0)), hp)


def test_random_layered_b64(g):
    p = W.random_layered(1)
    mu, sg = W.init_state(p, 64, 2)
    hp = g.default_hparams(terms=_cf(p.terms) | W.RES_VIOL, rho=1e-3)
    check_loss_grad(p, g, 64, mu, sg, _lam(64, np.random.default_rng(1)), hp, restarts=range(0, 64, 9))


def test_dep_cf_alone(g):
    p = W.random_layered(3)
    B = 8
    mu, sg = W.init_state(p, B, 3)
    hp = g.default_hparams(terms=W.DEP_CF, rho=1e-2)
    check_loss_grad(p, g, B, mu, sg, _lam(B, np.random.default_rng(5)), hp)


def test_modulo_with_recurrences_and_storage(g):
    p = W.modulo_loop(3, V=400, levels=20, n_back=20)
    terms = W.DEP_CF | W.RES_VIOL | W.REC | W.REG_OBJ
    mu, sg = W.init_state(p, 8, 4)
    hp = g.default_hparams(terms=terms, rho=1e-3)
    check_loss_grad(p, g, 8, mu, sg, _lam(8, np.random.default_rng(3)), hp)


def test_extreme_means_and_mixed_sigma(g):
    p = W.logic_network(6, V=1500, depth=30)
    B = 32
    rng = np.random.default_rng(12)
    mu = (p.start[:, None] + rng.normal(0, 2, size=(p.V, B))).astype(np.float32)
    sg = np.exp(rng.uniform(np.log(0.05), np.log(6.0), size=(p.V, B))).astype(np.float32)
    mu[3, 0], mu[4, 1] = -80.0, p.D + 80.0
    hp = g.default_hparams(terms=_cf(p.terms), rho=1e-3)
    check_loss_grad(p, g, B, mu, sg, _lam(B, rng), hp, restarts=range(0, 32, 4))


def test_logic_network_full_size_sampled(g):
    p = W.logic_network(1)
    mu, sg = W.init_state(p, 64, 1)
    hp = g.default_hparams(terms=_cf(p.terms))
    lam = np.full((64, 3), 1e-6, np.float32)
    check_loss_grad(p, g, 64, mu, sg, lam, hp, restarts=[0, 37])


def test_iterate_tracks_oracle_trajectory(g):
    p = W.tiny_layered(1)
    B = 2
    mu, sg = W.init_state(p, B, 1, mu_jitter="uniform01", sigma0=1.0)
    hp = g.default_hparams(terms=_cf(p.terms), lr=0.05)
    ctx = g.Gaus(p, B, hp)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=hp.tau, rho=hp.rho, alpha=hp.alpha, w_res=hp.w_res, w_mem=hp.w_mem,
                         terms=hp.terms)
    th_m, th_s = mu.astype(np.float64).copy(), sg.astype(np.float64).copy()
    mm = [np.zeros_like(th_m) for _ in range(4)]
    lam = np.full((B, 3), 1e-6)
    gl, ol = [], []
    for step in range(1, 21):
        ctx.iterate(1, st)
        loss, terms, gm, gs = oracle.loss_grad(op, ohp, th_m, th_s, lam)
        for b in range(B):
            for th, gg, m1, v1 in ((th_m, gm, mm[0], mm[1]), (th_s, gs, mm[2], mm[3])):
                col = np.ascontiguousarray(th[:, b])
                m_ = np.ascontiguousarray(m1[:, b]); v_ = np.ascontiguousarray(v1[:, b])
                oracle.adam(col, np.ascontiguousarray(gg[:, b]), m_, v_, step, hp.lr)
                th[:, b], m1[:, b], v1[:, b] = col, m_, v_
        th_s = np.maximum(th_s, hp.sigma_min)
        lam[:, 0] += hp.rho * terms[:, oracle.T_VDEP]
        lam[:, 1] += hp.rho * terms[:, oracle.T_VRES]
        torch.cuda.synchronize()
        gl.append(st["loss"].cpu().numpy().copy())
        ol.append(loss)
    gl, ol = np.array(gl), np.array(ol)
    np.testing.assert_allclose(gl[0], ol[0], rtol=1e-4)
    np.testing.assert_allclose(gl, ol, rtol=2e-2)
    ctx.close()
