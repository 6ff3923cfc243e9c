"""GPU path with the logistic, Laplace and Cauchy relaxations (App. D) against the
fp64 oracle, through the C ABI, with the tolerances of the normal's parity tests
(loss and terms 1e-4 relative + 1e-5; gradients 1e-4 of the restart's largest
component, and 1e-4 relative on every component above 1e-2 of it).

The heavier tails widen the windows: about 1.9x the normal's for the logistic,
2.4x for the Laplace, the whole horizon for the Cauchy, so these cases also run
the untabled and cooperative paths of the edge pass on every node.
"""
import numpy as np
import pytest

import oracle
import workloads as W

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from tests.test_gpu_parity import _lam, check_loss_grad  # noqa: E402

FAMS = [oracle.LOGISTIC, oracle.LAPLACE, oracle.CAUCHY]


@pytest.fixture(scope="module")
def g():
    import paper_2602_20427_gb300 as g
    g.build()
    g.lib()
    return g


@pytest.mark.parametrize("fam", FAMS)
def test_tiny_layered(g, fam):
    p = W.tiny_layered(1)
    B = 4
    mu, sg = W.init_state(p, B, 1, mu_jitter="uniform01", sigma0=1.0)
    hp = g.default_hparams(terms=p.terms, tau=0.05, rho=0.01, family=fam)
    check_loss_grad(p, g, B, mu, sg, _lam(B, np.random.default_rng(0)), hp)


@pytest.mark.parametrize("fam", FAMS)
def test_logic_small_all_terms(g, fam):
    p = W.logic_network(2, V=2000, depth=40)
    mu, sg = W.init_state(p, 32, 3)
    hp = g.default_hparams(terms=p.terms, alpha=0.7, w_res=1.3, rho=1e-3, family=fam)
    check_loss_grad(p, g, 32, mu, sg, _lam(32, np.random.default_rng(2)), hp, restarts=range(0, 32, 5))


@pytest.mark.parametrize("fam", FAMS)
def test_modulo_with_recurrences(g, fam):
    p = W.modulo_loop(3, V=400, levels=20, n_back=20)
    p.terms = W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL | W.REC
    mu, sg = W.init_state(p, 8, 4)
    hp = g.default_hparams(terms=p.terms, rho=1e-3, family=fam)
    check_loss_grad(p, g, 8, mu, sg, _lam(8, np.random.default_rng(3)), hp)


@pytest.mark.parametrize("fam", FAMS)
def test_storage_term(g, fam):
    p = W.random_small(31, V=40, D=30, C=2, max_lat=2, p_edge=0.12)
    p.terms = W.DEP | W.COM | W.REG_OBJ
    rng = np.random.default_rng(31)
    B = 8
    mu = (p.start[:, None] + rng.normal(0, 2, size=(p.V, B))).astype(np.float32)
    sg = rng.uniform(0.3, 2.5, size=(p.V, B)).astype(np.float32)
    hp = g.default_hparams(terms=p.terms, tau=0.3, w_mem=1.7, family=fam)
    check_loss_grad(p, g, B, mu, sg, _lam(B, rng), hp)


@pytest.mark.parametrize("fam", FAMS)
def test_storage_modulo(g, fam):
    p = W.modulo_loop(7, ii_factor=1.5, V=300, levels=15, n_back=15)
    p.terms = W.DEP | W.RES_VIOL | W.REG_OBJ | W.REC
    B = 8
    mu, sg = W.init_state(p, B, 12)
    hp = g.default_hparams(terms=p.terms, rho=1e-3, family=fam)
    check_loss_grad(p, g, B, mu, sg, _lam(B, np.random.default_rng(12)), hp, restarts=[0, 3, 7])


@pytest.mark.parametrize("fam", [oracle.GAUSSIAN] + FAMS)
def test_storage_small_tau(g, fam):
    # the loop body at full size (V = 5,000, D = 3 II = 1,659), where a folded step
    # sums hundreds of storage contributions, with tau = 3e-3 dividing their absolute
    # error by tau in the softmax weights: every family's tail table and Taylor step,
    # and the Cauchy series beyond the table (its windows span the horizon, z > 16),
    # against the oracle with the per-component bound from 1 % of the largest
    # component (test_modulo_loop_full_size_sampled_usage_and_storage is the normal's
    # case that contributions rounded to fp32 fail)
    p = W.modulo_loop(1, ii_factor=1.25)
    p.terms = W.RES_OBJ | W.RES_VIOL | W.REG_OBJ
    B = 8
    mu, sg = W.init_state(p, B, 13)
    hp = g.default_hparams(terms=p.terms, tau=3e-3, rho=1e-3, family=fam)
    lam = np.full((B, 3), 1e-6, np.float32)
    check_loss_grad(p, g, B, mu, sg, lam, hp, restarts=[0, 5])


@pytest.mark.parametrize("fam", FAMS)
def test_mixed_window_lengths(g, fam):
    # sigma over two orders of magnitude inside every warp
    p = W.logic_network(6, V=1500, depth=30)
    B = 32
    rng = np.random.default_rng(12)
    mu = (p.start[:, None] + rng.normal(0, 2, size=(p.V, B))).astype(np.float32)
    sg = np.exp(rng.uniform(np.log(0.05), np.log(6.0), size=(p.V, B))).astype(np.float32)
    hp = g.default_hparams(terms=p.terms, rho=1e-3, family=fam)
    check_loss_grad(p, g, B, mu, sg, _lam(B, rng), hp, restarts=range(0, 32, 4))


@pytest.mark.parametrize("fam", FAMS)
def test_means_outside_the_horizon_and_sigma_min(g, fam):
    p = W.random_layered(5)
    p.terms = W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL
    B = 6
    rng = np.random.default_rng(40 + fam)
    mu, sg = W.init_state(p, B, 5)
    mu[3, 0], mu[4, 1], mu[5, 2] = -50.0, p.D + 60.0, p.D - 0.50001
    sg[6, :] = 0.05
    sg[7:12, 3] = 9.0
    hp = g.default_hparams(terms=p.terms, tau=0.1, rho=0.01, family=fam)
    check_loss_grad(p, g, B, mu, sg, _lam(B, rng), hp)


def test_logistic_full_size_sampled(g):
    # the headline workload at its full size (V = 10,000, B = 64) with the
    # logistic relaxation; the oracle checks two restarts
    p = W.logic_network(1)
    mu, sg = W.init_state(p, 64, 1)
    hp = g.default_hparams(terms=p.terms, family=oracle.LOGISTIC)
    lam = np.full((64, 3), 1e-6, np.float32)
    check_loss_grad(p, g, 64, mu, sg, lam, hp, restarts=[0, 37])


def test_set_hparams_switches_the_family(g):
    # one context, the family switched in place, gives what a fresh context of
    # that family gives (bit for bit: same kernels, same inputs, fixed order)
    p = W.random_layered(2)
    B = 16
    mu, sg = W.init_state(p, B, 8)
    dmu, dsg = torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda()
    lam = torch.full((B, 3), 1e-6, device="cuda")
    outs = {}
    for fam in (oracle.GAUSSIAN, oracle.CAUCHY):
        ctx = g.Gaus(p, B, g.default_hparams(terms=p.terms, family=fam))
        outs[fam] = {k: v.clone() for k, v in ctx.loss_grad(dmu, dsg, lam).items()}
        ctx.close()
    ctx = g.Gaus(p, B, g.default_hparams(terms=p.terms))
    for fam in (oracle.CAUCHY, oracle.GAUSSIAN):
        ctx.set_hparams(g.default_hparams(terms=p.terms, family=fam))
        out = ctx.loss_grad(dmu, dsg, lam)
        torch.cuda.synchronize()
        for k in ("loss", "grad_mu", "grad_sigma"):
            assert torch.equal(out[k], outs[fam][k]), (fam, k)
    assert not torch.equal(outs[oracle.GAUSSIAN]["loss"], outs[oracle.CAUCHY]["loss"])
    ctx.close()


@pytest.mark.parametrize("path", ["fused", "multi"])
@pytest.mark.parametrize("fam", FAMS)
def test_iterate_tracks_oracle_trajectory(g, fam, path):
    # the iteration (loss, gradient, multipliers, Adam) on either path against the
    # oracle's loss per step on the tiny workload, gated as for the normal
    p = W.tiny_layered(1)
    B = 2
    mu, sg = W.init_state(p, B, 1, mu_jitter="uniform01", sigma0=1.0)
    hp = g.default_hparams(terms=p.terms, lr=0.05, family=fam)
    ctx = g.Gaus(p, B, hp)
    ctx.set_path(g.PATH_FUSED if path == "fused" else g.PATH_MULTI)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=hp.tau, rho=hp.rho, alpha=hp.alpha, w_res=hp.w_res, w_mem=hp.w_mem,
                         terms=p.terms, family=fam)
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
