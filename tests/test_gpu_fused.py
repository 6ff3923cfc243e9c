"""The persistent fused kernel's plan and its less common paths: the plan each term
set gets (gaus_plan_info), more restart groups than the device holds at once (one
cooperative launch per batch of groups), and the bounded group-barrier waits, whose
failure path is exercised with a barrier that nothing can complete (no fault, no
trap: the wait runs out and the restarts report GAUS_ETIMEOUT)."""
import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

from tests.test_gpu_parity import _lam, check_loss_grad  # noqa: E402

ETIMEOUT = 8


@pytest.fixture(scope="module")
def g():
    import paper_2602_20427_gb300 as g
    g.build()
    g.lib()
    return g


def test_plan_info_by_term_set(g):
    p = W.logic_network(3, V=1500, depth=30)
    B = 64
    # launches per iteration of the multi-kernel path: node, edge, reduce, finalize,
    # update, and the storage pass's three or the continuous penalty's one
    for terms, fused, per_iter in ((W.DEP | W.COM | W.RES_OBJ | W.RES_VIOL, 1, 5),
                                   (W.DEP | W.RES_VIOL | W.REG_OBJ, 0, 8),
                                   (W.DEP_CF | W.COM | W.RES_OBJ, 0, 6)):
        ctx = g.Gaus(p, B, g.default_hparams(terms=terms))
        info = ctx.plan_info()
        assert info["fused"] == fused, (terms, info)
        assert info["launches_per_iteration"] == per_iter, (terms, info)
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        assert info["sms"] == sms
        if fused:
            assert info["fused_launches_per_call"] == 1
            assert info["restart_groups"] == 1 and info["restarts_per_group"] == 64
            assert 1 <= info["blocks_per_group"] <= sms
            assert info["node_segments"] >= info["blocks_per_group"]
            assert 4 <= info["table_row_points"] <= 64
        ctx.close()


def test_more_restart_groups_than_resident(g):
    # 64 restarts per group, one more group than the device's SMs (one block per SM):
    # two cooperative launches per call, the last batch holding two groups, the very
    # last group ragged (5 restarts)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    p = W.tiny_layered(3)
    B = 64 * sms + 69
    mu, sg = W.init_state(p, B, 21, mu_jitter="uniform01", sigma0=1.0)
    hp = g.default_hparams(terms=p.terms, tau=0.05, rho=0.01)
    ctx = g.Gaus(p, B, hp)
    info = ctx.plan_info()
    assert info["fused"] == 1 and info["restart_groups"] == sms + 2
    assert info["fused_launches_per_call"] >= 2
    ctx.close()
    lam = _lam(B, np.random.default_rng(21))
    check_loss_grad(p, g, B, mu, sg, lam, hp, restarts=[0, 63, 64, 64 * sms, B - 1])
    # and the iteration: every restart's result equals the same restart run alone
    ctx = g.Gaus(p, B, hp)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    ctx.iterate(3, st)
    torch.cuda.synchronize()
    for b in (0, 64 * sms + 1, B - 1):
        one = g.Gaus(p, 1, hp)
        s1 = one.new_state(torch.from_numpy(mu[:, b:b + 1].copy()).cuda(),
                           torch.from_numpy(sg[:, b:b + 1].copy()).cuda(), 1e-6)
        one.iterate(3, s1)
        torch.cuda.synchronize()
        np.testing.assert_allclose(st["mu"][:, b].cpu().numpy(), s1["mu"][:, 0].cpu().numpy(), rtol=0, atol=1e-6)
        np.testing.assert_allclose(st["sigma"][:, b].cpu().numpy(), s1["sigma"][:, 0].cpu().numpy(), rtol=0,
                                   atol=1e-6)
        np.testing.assert_allclose(st["loss"][b].item(), s1["loss"][0].item(), rtol=1e-6)
        one.close()
    assert np.all(st["status"].cpu().numpy() == 0)
    ctx.close()


def test_barrier_wait_runs_out_and_reports(g):
    # a group barrier that no block can complete: each wait ends after 2 ms, every
    # restart reports GAUS_ETIMEOUT, the caller's state is untouched, and the same
    # context then iterates as a fresh one does (up to the lane each restart lands on:
    # the aborted call left its own restart order behind)
    p = W.random_layered(2)
    B = 96  # two restart groups
    mu, sg = W.init_state(p, B, 2)
    hp = g.default_hparams(terms=p.terms)
    ctx = g.Gaus(p, B, hp)
    st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    before = {k: v.clone() for k, v in st.items()}
    ctx.check_barrier_timeout(st, 2_000_000)
    torch.cuda.synchronize()
    assert np.all(st["status"].cpu().numpy() == ETIMEOUT)
    for k in ("mu", "sigma", "m_mu", "v_mu", "m_sigma", "v_sigma", "lambda_", "step"):
        assert torch.equal(st[k], before[k]), k
    st["status"].zero_()
    ctx.iterate(2, st)
    fresh = g.Gaus(p, B, hp)
    s2 = fresh.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
    fresh.iterate(2, s2)
    torch.cuda.synchronize()
    assert np.all(st["status"].cpu().numpy() == 0)
    for k in ("mu", "sigma", "lambda_", "loss"):
        np.testing.assert_allclose(st[k].cpu().numpy(), s2[k].cpu().numpy(), rtol=1e-6, atol=1e-6, err_msg=k)
    fresh.close()
    # the multi-kernel path has no group barriers
    reg = g.Gaus(p, B, g.default_hparams(terms=p.terms | W.REG_OBJ))
    with pytest.raises(g.GausError):
        reg.check_barrier_timeout(reg.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda()), 2_000_000)
    reg.close()
    ctx.close()


def test_auto_path_choice(g):
    # GAUS_PATH_AUTO per call: the fused kernel for uniform windows within its staging
    # (sigma = 1.5: about 18 points everywhere) and for windows under a point on
    # average (sigma = 0.1); the multi-kernel path for windows that vary across
    # restarts (sigma from 0.2 to 3) and for windows beyond the staging (logistic,
    # about 34 points at sigma = 1.5); the forced modes whatever the windows
    p = W.logic_network(4, V=2000, depth=40)
    B = 64
    rng = np.random.default_rng(5)
    mu, _ = W.init_state(p, B, 5)
    cases = (("uniform", g.GAUSSIAN, np.full((p.V, B), 1.5, np.float32), "fused"),
             ("short", g.GAUSSIAN, np.full((p.V, B), 0.1, np.float32), "fused"),
             ("varied", g.GAUSSIAN, rng.uniform(0.2, 3.0, size=(p.V, B)).astype(np.float32), "multi"),
             ("wide tails", g.LOGISTIC, np.full((p.V, B), 1.5, np.float32), "multi"))
    for name, fam, sg, want in cases:
        ctx = g.Gaus(p, B, g.default_hparams(terms=p.terms, family=fam))
        st = ctx.new_state(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), 1e-6)
        i0 = ctx.plan_info()
        ctx.iterate(3, st)
        torch.cuda.synchronize()
        i1 = ctx.plan_info()
        got = "fused" if i1["fused_calls"] - i0["fused_calls"] == 1 else "multi"
        assert got == want, (name, i0, i1)
        assert i1["path_choices"] - i0["path_choices"] == 1
        assert i1["multi_iterations"] - i0["multi_iterations"] == (3 if want == "multi" else 0)
        for mode, forced in ((g.PATH_FUSED, "fused"), (g.PATH_MULTI, "multi")):
            ctx.set_path(mode)
            j0 = ctx.plan_info()
            ctx.iterate(2, st)
            j1 = ctx.plan_info()
            assert j1["path_mode"] == mode and j1["path_choices"] == j0["path_choices"]
            assert (j1["fused_calls"] - j0["fused_calls"]) == (1 if forced == "fused" else 0), (name, mode)
        torch.cuda.synchronize()
        assert np.all(st["status"].cpu().numpy() == 0)
        ctx.close()
    # decided by the sizes, with no reduction: a tiny problem (64 nodes, one restart)
    # runs the fused kernel, restart groups of 16 the multi-kernel path
    for pp, BB, want in ((W.tiny_layered(1), 1, "fused"), (p, 16, "multi")):
        mu_s, sg_s = W.init_state(pp, BB, 7)
        c = g.Gaus(pp, BB, g.default_hparams(terms=pp.terms))
        st = c.new_state(torch.from_numpy(mu_s).cuda(), torch.from_numpy(sg_s).cuda(), 1e-6)
        c.iterate(2, st)
        torch.cuda.synchronize()
        i1 = c.plan_info()
        assert i1["path_choices"] == 0
        assert (i1["fused_calls"], i1["multi_iterations"]) == ((1, 0) if want == "fused" else (0, 2)), (BB, i1)
        c.close()
    with pytest.raises(g.GausError):
        c = g.Gaus(p, B, g.default_hparams(terms=p.terms))
        try:
            c.set_path(3)
        finally:
            c.close()
