"""Rounding, legalization (Alg. 1, Alg. 2), verification, Adam and the fused
iteration on the GPU against the oracle.  Integer results are bit-exact."""
import numpy as np
import pytest

import oracle
import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def g():
    import paper_2602_20427_gb300 as g
    g.build()
    g.lib()
    return g


def test_round_half_up_exact(g):
    p = W.tiny_layered(1)
    B = 4
    vals = np.array([-1.5, -0.5, -0.49999997, 0.0, 0.49999997, 0.5, 1.5, 2.4999998, 7.5, 1e7 + 0.5],
                    dtype=np.float32)
    mu = np.resize(vals, (p.V, B)).astype(np.float32)
    ctx = g.Gaus(p, B)
    s = ctx.round(torch.from_numpy(mu).cuda()).cpu().numpy()
    np.testing.assert_array_equal(s, oracle.round_half_up(mu.astype(np.float64)))
    ctx.close()


def _legalize_and_verify(g, p, B, mu):
    ctx = g.Gaus(p, B)
    dmu = torch.from_numpy(mu).cuda()
    sched, status = ctx.legalize(dmu)
    reps = ctx.verify(sched)
    raw = ctx.verify(ctx.round(dmu))
    torch.cuda.synchronize()
    a_asap, a_alap, a_cp = ctx.bounds()
    ctx.close()
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    np.testing.assert_array_equal(a_asap, asap)
    np.testing.assert_array_equal(a_alap, alap)
    assert a_cp == cp
    s_np, st_np = sched.cpu().numpy(), status.cpu().numpy()
    for b in range(B):
        s0 = oracle.round_half_up(mu[:, b].astype(np.float64))
        if p.II > 0:
            ref, rc2 = oracle.legalize_modulo(op, order, s0)
            assert st_np[b] == (7 if rc2 else 0)
            if rc2:
                continue            # unsettled: the schedule is unspecified
        else:
            ref = oracle.legalize_regular(op, order, asap, alap, s0)
            assert st_np[b] == 0
        np.testing.assert_array_equal(s_np[:, b], ref)
        r = oracle.verify(op, ref)
        for k in oracle.REPORT_FIELDS:
            assert reps[b][k] == r[k], (b, k)
        assert reps[b]["peak"] == r["peak"]
        r0 = oracle.verify(op, s0)
        for k in oracle.REPORT_FIELDS:
            assert raw[b][k] == r0[k], (b, k, "raw")


def test_legalize_verify_regular_random(g):
    p = W.random_layered(3)
    mu, _ = W.init_state(p, 64, 3)
    _legalize_and_verify(g, p, 64, mu)


def test_legalize_verify_regular_logic(g):
    p = W.logic_network(4, V=3000, depth=50)
    mu, _ = W.init_state(p, 32, 4)
    _legalize_and_verify(g, p, 32, mu)


@pytest.mark.parametrize("factor", [1.0, 1.5])
def test_legalize_verify_modulo(g, factor):
    p = W.modulo_loop(5, ii_factor=factor, V=600, levels=20, n_back=30)
    mu, _ = W.init_state(p, 16, 5)
    _legalize_and_verify(g, p, 16, mu)


def test_legalize_verify_regular_global_memory_path(g):
    # V = 60,000: a schedule (4 V bytes) no longer fits one block's shared memory, so
    # Alg. 1 runs in its global-memory form
    p = W.wide_layered(2, width=1200, levels=50)
    mu, _ = W.init_state(p, 3, 2)
    _legalize_and_verify(g, p, 3, mu)


def test_legalize_verify_modulo_full_size(g):
    # the loop-body workload at its full size (V = 5,000, 200 back edges, B = 32)
    p = W.modulo_loop(1, ii_factor=1.25)
    mu, _ = W.init_state(p, 32, 1)
    _legalize_and_verify(g, p, 32, mu)


def test_legalize_modulo_reports_infeasible_recurrence(g):
    p = W.random_small(5, V=6, D=12, p_edge=1.0, max_lat=1)
    p.lat[:] = 1
    p.bsrc = np.array([5], np.int32)
    p.bdst = np.array([0], np.int32)
    p.bdist = np.array([1], np.int32)
    p.II = 2
    mu = np.zeros((6, 3), np.float32)
    ctx = g.Gaus(p, 3)
    sched, status = ctx.legalize(torch.from_numpy(mu).cuda())
    torch.cuda.synchronize()
    assert np.all(status.cpu().numpy() == 7)
    ctx.close()


def test_adam_step_matches_oracle(g):
    p = W.random_layered(1)
    B = 16
    rng = np.random.default_rng(0)
    mu, sg = W.init_state(p, B, 1)
    hp = g.default_hparams(terms=p.terms)
    ctx = g.Gaus(p, B, hp)
    t = {k: torch.from_numpy(v).cuda() for k, v in (("mu", mu), ("sg", sg))}
    z = [torch.zeros((p.V, B), device="cuda") for _ in range(4)]
    lam = torch.full((B, 3), 1e-6, device="cuda")
    th = [mu.astype(np.float64).ravel().copy(), sg.astype(np.float64).ravel().copy()]
    mo = [np.zeros(p.V * B) for _ in range(4)]
    # the multiplier update of Sec. 3.3, lambda_k <- lambda_k + rho V_k for every active
    # constraint k (dependency, resource excess, recurrence), others unchanged
    lam_ref = np.full((B, 3), 1e-6)
    active = [(oracle.K_DEP, oracle.T_VDEP, bool(p.terms & W.DEP)),
              (oracle.K_RES, oracle.T_VRES, bool(p.terms & W.RES_VIOL)),
              (oracle.K_REC, oracle.T_VREC, bool(p.terms & W.REC))]
    assert any(a for _, _, a in active)
    for step in range(1, 4):
        gm = (rng.normal(size=(p.V, B)) * 10 ** rng.uniform(-3, 1)).astype(np.float32)
        gs = (rng.normal(size=(p.V, B)) * 10 ** rng.uniform(-3, 1)).astype(np.float32)
        T = rng.uniform(0, 5, size=(B, 6)).astype(np.float32)
        terms = torch.from_numpy(T).cuda()
        ctx.adam_step(t["mu"], t["sg"], torch.from_numpy(gm).cuda(), torch.from_numpy(gs).cuda(), *z, lam,
                      terms, step)
        oracle.adam(th[0], gm.astype(np.float64).ravel().copy(), mo[0], mo[1], step, hp.lr)
        oracle.adam(th[1], gs.astype(np.float64).ravel().copy(), mo[2], mo[3], step, hp.lr)
        th[1] = np.maximum(th[1], hp.sigma_min)
        for k, tk, on in active:
            if on:
                lam_ref[:, k] += hp.rho * T[:, tk].astype(np.float64)
        torch.cuda.synchronize()
        np.testing.assert_allclose(lam.cpu().numpy(), lam_ref, rtol=1e-6, atol=0)
    torch.cuda.synchronize()
    np.testing.assert_allclose(t["mu"].cpu().numpy().ravel(), th[0], rtol=0, atol=2e-5)
    np.testing.assert_allclose(t["sg"].cpu().numpy().ravel(), th[1], rtol=0, atol=2e-5)
    ctx.close()


@pytest.mark.parametrize("path", ["fused", "multi"])
def test_iterate_equals_separate_calls(g, path):
    # the iteration computes the same as loss_grad + adam_step, on either path
    p = W.random_layered(2)
    B = 32
    mu, sg = W.init_state(p, B, 2)
    hp = g.default_hparams(terms=p.terms)
    ctx = g.Gaus(p, B, hp)
    ctx.set_path(g.PATH_FUSED if path == "fused" else g.PATH_MULTI)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    m = {k: torch.from_numpy(v).cuda() for k, v in (("mu", mu), ("sg", sg))}
    z = [torch.zeros((p.V, B), device="cuda") for _ in range(4)]
    lam = torch.full((B, 3), 1e-6, device="cuda")
    for step in range(1, 6):
        ctx.iterate(1, st)
        out = ctx.loss_grad(m["mu"], m["sg"], lam)
        ctx.adam_step(m["mu"], m["sg"], out["grad_mu"], out["grad_sigma"], *z, lam, out["terms"], step)
        torch.cuda.synchronize()
        np.testing.assert_allclose(st["loss"].cpu().numpy(), out["loss"].cpu().numpy(), rtol=1e-5)
    np.testing.assert_allclose(st["mu"].cpu().numpy(), m["mu"].cpu().numpy(), rtol=0, atol=1e-4)
    np.testing.assert_allclose(st["sigma"].cpu().numpy(), m["sg"].cpu().numpy(), rtol=0, atol=1e-4)
    np.testing.assert_allclose(st["lambda_"].cpu().numpy(), lam.cpu().numpy(), rtol=1e-5)
    assert np.all(st["step"].cpu().numpy() == 5)
    ctx.close()


@pytest.mark.parametrize("path", ["fused", "multi"])
def test_iterate_multiplier_update(g, path):
    # the iteration's multiplier update (Sec. 3.3), on either path: after every iteration,
    # lambda_k = lambda_k(before) + rho V_k for the active constraints, with V_k the
    # values the iteration reports (exactly, up to the final rounding to float) and
    # against the oracle's V_k at the same state (within the parity tolerance)
    p = W.random_layered(3)
    p.terms = W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL
    B = 8
    mu, sg = W.init_state(p, B, 3)
    hp = g.default_hparams(terms=p.terms, rho=1e-2)
    ctx = g.Gaus(p, B, hp)
    ctx.set_path(g.PATH_FUSED if path == "fused" else g.PATH_MULTI)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-3)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=hp.tau, rho=hp.rho, alpha=hp.alpha, w_res=hp.w_res, w_mem=hp.w_mem, terms=p.terms)
    for it in range(4):
        lam0 = st["lambda_"].cpu().numpy().astype(np.float64)
        m0 = st["mu"].cpu().numpy().astype(np.float64)
        s0 = st["sigma"].cpu().numpy().astype(np.float64)
        ctx.iterate(1, st)
        torch.cuda.synchronize()
        lam1 = st["lambda_"].cpu().numpy().astype(np.float64)
        T = st["terms"].cpu().numpy().astype(np.float64)
        own = lam0.copy()
        own[:, oracle.K_DEP] += hp.rho * T[:, oracle.T_VDEP]
        own[:, oracle.K_RES] += hp.rho * T[:, oracle.T_VRES]
        np.testing.assert_allclose(lam1, own, rtol=2e-7, atol=0)
        assert np.all(lam1[:, oracle.K_REC] == lam0[:, oracle.K_REC])
        _, Tref, _, _ = oracle.loss_grad(op, ohp, m0, s0, lam0)
        ref = lam0.copy()
        ref[:, oracle.K_DEP] += hp.rho * Tref[:, oracle.T_VDEP]
        ref[:, oracle.K_RES] += hp.rho * Tref[:, oracle.T_VRES]
        np.testing.assert_allclose(lam1 - lam0, ref - lam0, rtol=1e-4, atol=2e-5 * hp.rho)
    ctx.close()


@pytest.mark.parametrize("path", ["fused", "multi"])
def test_iterate_tracks_oracle_trajectory(g, path):
    # a short trajectory of the tiny workload against the oracle, on either path
    # (reported quantity: the loss per step; gated loosely because first-step Adam is
    # sign-like and can flip noise-level components)
    p = W.tiny_layered(1)
    B = 2
    mu, sg = W.init_state(p, B, 1, mu_jitter="uniform01", sigma0=1.0)
    hp = g.default_hparams(terms=p.terms, lr=0.05)
    ctx = g.Gaus(p, B, hp)
    ctx.set_path(g.PATH_FUSED if path == "fused" else g.PATH_MULTI)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=hp.tau, rho=hp.rho, alpha=hp.alpha, w_res=hp.w_res, w_mem=hp.w_mem, terms=p.terms)
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


def test_two_live_contexts_of_different_sizes(g):
    # kernel launch limits are per process: a second, smaller context must not break
    # the first one's launches (legalize, verify, iterate interleaved)
    big, small = W.random_layered(1), W.tiny_layered(1)
    ctxs = []
    for p, B in ((big, 16), (small, 4)):
        c = g.Gaus(p, B, g.default_hparams(terms=p.terms))
        mu, sg = W.init_state(p, B, 1)
        st = c.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
        ctxs.append((c, st, p))
    for c, st, p in ctxs * 2:
        c.iterate(2, st)
        sched, status = c.legalize(st["mu"])
        c.verify(sched)
        torch.cuda.synchronize()
        assert np.all(status.cpu().numpy() == 0)
    for c, _, _ in ctxs:
        c.close()
