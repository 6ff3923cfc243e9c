"""gaus_expected_usage_noalloc: the usage reduction for callers that cannot
allocate device memory, checked against the context-based entry point.

gaus_loss_grad reports, per restart, the sum over classes of LSE_tau(usage) and
the summed ReLU excess over the limits; both are recomputed here (float64) from
the usage that the allocation-free entry point writes, and must agree within the
tolerance of the other parity tests, on two calls in a row (with different
inputs, so that nothing left in the shared scratch array can leak through).
The file is collected last on purpose: a failure here cannot hide another test.
"""
import ctypes as C

import numpy as np
import pytest
from scipy.special import logsumexp

import oracle
import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

T_RES, T_VRES = 0, 4   # columns of the per-restart term values (include/gaus.h)


@pytest.fixture(scope="module")
def g():
    import paper_2602_20427_gb300 as g
    g.build()
    g.lib()
    return g


def _usage(g, p, mu, sg, window_k):
    dev = torch.device("cuda")
    Dh = p.II if p.II > 0 else p.D
    out = torch.full((mu.shape[1], p.C, Dh), -1.0, dtype=torch.float64, device=dev)
    t = [torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in
         (mu, sg, np.asarray(p.cls, np.int32), np.asarray(p.demand, np.int32))]
    rc = g.lib().gaus_expected_usage_noalloc(
        C.c_void_p(t[0].data_ptr()), C.c_void_p(t[1].data_ptr()), C.c_void_p(t[2].data_ptr()),
        C.c_void_p(t[3].data_ptr()), C.c_int32(p.V), C.c_int32(mu.shape[1]), C.c_int32(p.C), C.c_int32(p.D),
        C.c_int32(p.II), C.c_float(window_k), C.c_void_p(out.data_ptr()),
        C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0, g.lib().gaus_last_error(None)
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("which", ["logic", "modulo"])
def test_usage_noalloc_matches_loss_grad_on_two_calls(g, which):
    if which == "logic":
        p = W.logic_network(2, V=2000, depth=40)
    else:
        p = W.modulo_loop(3, V=400, levels=20, n_back=20)
    B = 32
    terms = W.RES_OBJ | W.RES_VIOL
    hp = g.default_hparams(terms=terms)
    ctx = g.Gaus(p, B, hp)
    lam = torch.full((B, 3), 1e-6, device="cuda")
    for call in range(2):
        mu, sg = W.init_state(p, B, seed=40 + call)
        U = _usage(g, p, mu, sg, hp.window_k)
        out = ctx.loss_grad(torch.from_numpy(mu).cuda(), torch.from_numpy(sg).cuda(), lam)
        T = out["terms"].cpu().numpy()
        lse = np.array([sum(hp.tau * logsumexp(U[b, c] / hp.tau) for c in range(p.C)) for b in range(B)])
        lim = np.asarray(p.limit, np.float64)
        relu = np.array([sum(np.maximum(U[b, c] - lim[c], 0).sum() for c in range(p.C) if np.isfinite(lim[c]))
                         for b in range(B)])
        np.testing.assert_allclose(lse, T[:, T_RES], rtol=1e-4, atol=1e-5)
        np.testing.assert_allclose(relu, T[:, T_VRES], rtol=1e-4, atol=1e-5)
        # and the usage itself against the fp64 oracle for two restarts
        op = oracle.OracleProblem(p)
        for b in (0, B - 1):
            ref, _ = oracle.expected_hist(op, mu[:, b].astype(np.float64), sg[:, b].astype(np.float64))
            np.testing.assert_allclose(U[b], ref, rtol=1e-5, atol=1e-5)
    ctx.close()


def test_usage_noalloc_rejects_oversized_problems(g):
    p = W.logic_network(2, V=2000, depth=40)
    mu, sg = W.init_state(p, 32, seed=3)
    d = torch.zeros(1, device="cuda")
    # a histogram length beyond the documented limit: nothing is launched
    rc = g.lib().gaus_expected_usage_noalloc(
        C.c_void_p(d.data_ptr()), C.c_void_p(d.data_ptr()), C.c_void_p(d.data_ptr()), None,
        C.c_int32(10), C.c_int32(32), C.c_int32(2), C.c_int32(2000), C.c_int32(0), C.c_float(6.0),
        C.c_void_p(d.data_ptr()), None)
    assert rc == 1
    assert b"25,600" in g.lib().gaus_last_error(None)
