"""The C-ABI library builds, loads and exports every entry point of include/gaus.h;
host-side validation of gaus_create runs without a GPU (no compute calls)."""
import ctypes as C
import math
import shutil

import numpy as np
import pytest

import paper_2602_20427_gb300 as g
import workloads as W

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not __import__("os").path.exists(
    "/usr/local/cuda/bin/nvcc"), reason="nvcc not available")


@pytest.fixture(scope="module")
def L():
    g.build()
    return g.lib()


def test_every_declared_symbol_is_exported(L):
    names = g.symbols_declared()
    assert len(names) >= 12
    for n in names:
        assert hasattr(L, n), n


def test_default_hparams_are_the_paper_values(L):
    h = g.default_hparams()
    assert h.tau == pytest.approx(1e-2) and h.rho == pytest.approx(1e-4)
    assert h.lambda0 == pytest.approx(1e-6) and h.lr == pytest.approx(1e-2)
    assert (h.beta1, h.beta2) == (pytest.approx(0.9), pytest.approx(0.999))
    assert h.terms == g.DEP | g.COM | g.RES_OBJ
    assert h.family == g.GAUSSIAN
    assert L.gaus_default_hparams(None) == 1


def _problem(p, B=2):
    keep = []

    def arr(x, dt):
        a = np.ascontiguousarray(np.asarray(x, dt))
        keep.append(a)
        return a.ctypes.data if a.size else None

    src, dst = np.asarray(p.src, np.int64), np.asarray(p.dst, np.int64)
    sp, si = g._csr(p.V, src, dst)
    pp, pi = g._csr(p.V, dst, src)
    pr = g.Problem(p.V, src.size, arr(sp, np.int32), arr(si, np.int32), arr(pp, np.int32), arr(pi, np.int32),
                   arr(p.lat, np.int32), arr(p.cls, np.int32), p.C, arr(p.limit, np.float32),
                   arr(p.demand, np.int32), arr(p.bits, np.int32), int(np.asarray(p.bsrc).size),
                   arr(p.bsrc, np.int32), arr(p.bdst, np.int32), arr(p.bdist, np.int32), p.D, p.II, B)
    return pr, keep


def _create(L, pr, hp=None):
    hp = hp or g.default_hparams()
    ctx = C.c_void_p()
    rc = L.gaus_create(C.byref(pr), C.byref(hp), None, C.byref(ctx))
    msg = L.gaus_last_error(None).decode()
    if rc == 0:
        L.gaus_destroy(ctx)
    return rc, msg


def test_create_validation_errors_without_gpu(L):
    p = W.tiny_layered(1)
    pr, keep = _problem(p)
    # a cycle
    q = W.random_small(1, V=4, D=8, p_edge=0.0)
    q.src = np.array([0, 1, 2], np.int32)
    q.dst = np.array([1, 2, 0], np.int32)
    pq, k2 = _problem(q)
    assert _create(L, pq)[0] == 2
    # horizon shorter than the critical path
    p2 = W.tiny_layered(1)
    p2.D = p2.cp - 1
    ph, k3 = _problem(p2)
    assert _create(L, ph)[0] == 3
    # bad class count, bad B, bad D
    for field, val in (("C", 0), ("B", 0), ("D", 0), ("II", -1)):
        bad, k4 = _problem(p)
        setattr(bad, field, val)
        assert _create(L, bad)[0] == 1, field
    # CSR and CSC that disagree
    bad, k5 = _problem(p)
    pi = np.ctypeslib.as_array(C.cast(bad.pred_idx, C.POINTER(C.c_int32)), shape=(p.E,))
    pi[0] = (pi[0] + 1) % p.V
    assert _create(L, bad)[0] == 1
    # REC without II
    hp = g.default_hparams(terms=g.DEP | g.REC)
    assert _create(L, pr, hp)[0] == 1
    # hparams out of range
    assert _create(L, pr, g.default_hparams(tau=0.0))[0] == 1
    assert _create(L, pr, g.default_hparams(beta1=1.0))[0] == 1
    assert _create(L, pr, g.default_hparams(family=4))[0] == 1
    assert _create(L, pr, g.default_hparams(family=-1))[0] == 1
    # the two forms of the dependency constraint exclude each other; the closed form is the normal's
    assert _create(L, pr, g.default_hparams(terms=g.DEP | g.DEP_CF))[0] == 1
    assert _create(L, pr, g.default_hparams(terms=g.DEP_CF, family=g.LOGISTIC))[0] == 1
    assert _create(L, pr, g.default_hparams(terms=128))[0] == 1


def test_valid_problem_reaches_the_device_check(L):
    import torch
    if torch.cuda.is_available():
        pytest.skip("GPU present: covered by the GPU tests")
    pr, keep = _problem(W.tiny_layered(1))
    rc, msg = _create(L, pr)
    assert rc == 5 and "CUDA" in msg


def test_measure_peak_rejects_bad_arguments_without_gpu(L):
    import ctypes as C
    v = C.c_double()
    assert L.gaus_measure_peak(C.c_int32(7), C.byref(v), None) == 1
    assert L.gaus_measure_peak(C.c_int32(g.PEAK_FP32), None, None) == 1
