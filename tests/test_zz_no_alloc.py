"""gaus_expected_usage_noalloc: the usage reduction for callers that cannot
allocate device memory, checked against the context-based entry point.

gaus_loss_grad reports, per restart, the sum over classes of LSE_tau(usage) and
the summed ReLU excess over the limits; both are recomputed here (float64) from
the usage that the allocation-free entry point writes, and must agree within the
tolerance of the other parity tests, on two calls in a row (with different
inputs, so that nothing left in the shared scratch array can leak through).  The
usage itself is checked against the fp64 oracle for several row widths, restart
groups and demands, and a demand beyond the histogram's bound must show as NaN.
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


def _usage(g, p, mu, sg, window_k, demand=True):
    """Call the entry point; demand=False passes NULL (every demand 1)."""
    dev = torch.device("cuda")
    Dh = p.II if p.II > 0 else p.D
    out = torch.full((mu.shape[1], p.C, Dh), -1.0, dtype=torch.float64, device=dev)
    t = [torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in
         (mu, sg, np.asarray(p.cls, np.int32), np.asarray(p.demand, np.int32))]
    rc = g.lib().gaus_expected_usage_noalloc(
        C.c_void_p(t[0].data_ptr()), C.c_void_p(t[1].data_ptr()), C.c_void_p(t[2].data_ptr()),
        C.c_void_p(t[3].data_ptr()) if demand else None, C.c_int32(p.V), C.c_int32(mu.shape[1]),
        C.c_int32(p.C), C.c_int32(p.D), C.c_int32(p.II), C.c_float(window_k), C.c_void_p(out.data_ptr()),
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


@pytest.mark.parametrize("B", [5, 40])
@pytest.mark.parametrize("demand", ["null", "seeded"])
def test_usage_noalloc_rows_groups_and_demands(g, B, demand):
    # B = 5: rows of 8 restarts, four nodes per warp sharing shared-memory cells;
    # B = 40: two restart groups with their own completion counters; demands NULL
    # (every demand 1) or seeded integers in 1..64, against the fp64 oracle with the
    # same demands, on two calls in a row
    p = W.modulo_loop(5, V=300, levels=15, n_back=10)
    rng = np.random.default_rng(70 + B)
    if demand == "seeded":
        p.demand = rng.integers(1, 65, size=p.V).astype(np.int32)
    else:
        p.demand = np.ones(p.V, np.int32)
    op = oracle.OracleProblem(p)
    for call in range(2):
        mu, sg = W.init_state(p, B, seed=80 + call)
        U = _usage(g, p, mu, sg, 6.0, demand=(demand == "seeded"))
        for b in sorted({0, B // 2, B - 1}):
            ref, _ = oracle.expected_hist(op, mu[:, b].astype(np.float64), sg[:, b].astype(np.float64))
            np.testing.assert_allclose(U[b], ref, rtol=1e-5, atol=1e-5 * max(1.0, float(p.demand.max())))


def test_usage_noalloc_flags_a_demand_above_64(g):
    # a demand the fixed-point histogram cannot hold (65) is not added: the rows of
    # its class become NaN for every restart, the other classes' rows are unaffected
    p = W.logic_network(2, V=2000, depth=40)
    B = 8
    v = int(np.flatnonzero(np.asarray(p.cls) == 0)[5])
    p.demand = np.ones(p.V, np.int32)
    p.demand[v] = 65
    mu, sg = W.init_state(p, B, seed=90)
    U = _usage(g, p, mu, sg, 6.0)
    assert np.all(np.isnan(U[:, 0, :]))
    assert np.all(np.isfinite(U[:, 1, :]))
    op = oracle.OracleProblem(p)
    ref, _ = oracle.expected_hist(op, mu[:, 3].astype(np.float64), sg[:, 3].astype(np.float64))
    np.testing.assert_allclose(U[3, 1], ref[1], rtol=1e-5, atol=1e-5)


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
