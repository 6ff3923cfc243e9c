"""fp64 CPU oracle for GauS (arXiv 2602.20427) -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` import this package.  It wraps ``gaus_oracle.c`` (plain C, built
with gcc into ``oracle/_build/liboracle.so``) and shares no code with the CUDA
library.  Per-restart arrays cross this wrapper in the (V, B) layout that the
library uses; the C side works restart-major.

Every function cites the passage of the paper it follows in ``gaus_oracle.c``.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gaus_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")

DEP, COM, RES_OBJ, RES_VIOL, REG_OBJ, REC = 1, 2, 4, 8, 16, 32
# not the paper's Eq. dep: sum_e Phi((mu_u + Lat(u) - mu_v) / sqrt(sigma_u^2 + sigma_v^2)),
# the continuous dependency penalty, a variant with the same multiplier as DEP
DEP_CF = 64
K_DEP, K_RES, K_REC, K = 0, 1, 2, 3
T_RES, T_COM, T_REG, T_VDEP, T_VRES, T_VREC, NT = 0, 1, 2, 3, 4, 5, 6
# CDF families of the relaxation (Sec. 3.2; App. D)
GAUSSIAN, LOGISTIC, LAPLACE, CAUCHY = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp64, OpenMP over restarts)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    hdr = os.path.join(_HERE, "gaus_oracle.h")
    if not force and os.path.exists(_LIB) and \
            os.path.getmtime(_LIB) >= max(os.path.getmtime(_SRC), os.path.getmtime(hdr)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-D_DEFAULT_SOURCE", "-fopenmp", "-fPIC",
                    "-shared", "-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, _LIB)
    return _LIB


class _Problem(C.Structure):
    _fields_ = [("V", C.c_int32), ("E", C.c_int32),
                ("src", C.c_void_p), ("dst", C.c_void_p), ("lat", C.c_void_p),
                ("cls", C.c_void_p), ("C", C.c_int32), ("limit", C.c_void_p),
                ("demand", C.c_void_p), ("bits", C.c_void_p), ("NB", C.c_int32),
                ("bsrc", C.c_void_p), ("bdst", C.c_void_p), ("bdist", C.c_void_p),
                ("D", C.c_int32), ("II", C.c_int32)]


class _Hparams(C.Structure):
    _fields_ = [("tau", C.c_double), ("rho", C.c_double), ("alpha", C.c_double),
                ("w_res", C.c_double), ("w_mem", C.c_double), ("terms", C.c_uint32),
                ("family", C.c_int32)]


class _Report(C.Structure):
    _fields_ = [("n_dep_viol", C.c_int64), ("n_lat_viol", C.c_int64),
                ("n_rec_viol", C.c_int64), ("n_res_viol", C.c_int64),
                ("L_res", C.c_int64), ("L_com", C.c_int64), ("L_mem", C.c_int64),
                ("L_mmem", C.c_int64), ("peak", C.c_int64 * 16),
                ("feasible", C.c_int32), ("res_ok", C.c_int32)]


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        _lib.orc_Phi.restype = C.c_double
        _lib.orc_Phi.argtypes = [C.c_double]
        _lib.orc_phi.restype = C.c_double
        _lib.orc_phi.argtypes = [C.c_double]
        _lib.orc_F.restype = C.c_double
        _lib.orc_F.argtypes = [C.c_int32, C.c_double]
        _lib.orc_f.restype = C.c_double
        _lib.orc_f.argtypes = [C.c_int32, C.c_double]
        _lib.orc_asap_alap.restype = C.c_int
        _lib.orc_legalize_modulo.restype = C.c_int
        _lib.orc_outer_step.restype = C.c_int32
    return _lib


def _p(a):
    return C.c_void_p(a.ctypes.data)


class OracleProblem:
    """Holds contiguous copies of a problem's arrays and the C view of them."""

    def __init__(self, prob):
        self.V, self.E, self.C, self.D, self.II = prob.V, prob.E, prob.C, prob.D, prob.II
        i32 = lambda x: np.ascontiguousarray(np.asarray(x, dtype=np.int32))
        f64 = lambda x: np.ascontiguousarray(np.asarray(x, dtype=np.float64))
        self.src, self.dst = i32(prob.src), i32(prob.dst)
        self.lat, self.cls = i32(prob.lat), i32(prob.cls)
        self.limit, self.demand, self.bits = f64(prob.limit), f64(prob.demand), f64(prob.bits)
        self.bsrc, self.bdst, self.bdist = i32(prob.bsrc), i32(prob.bdst), i32(prob.bdist)
        self.NB = int(self.bsrc.size)
        self.c = _Problem(self.V, self.E, _p(self.src).value, _p(self.dst).value,
                          _p(self.lat).value, _p(self.cls).value, self.C,
                          _p(self.limit).value, _p(self.demand).value, _p(self.bits).value,
                          self.NB, _p(self.bsrc).value, _p(self.bdst).value,
                          _p(self.bdist).value, self.D, self.II)

    @property
    def Dh(self):
        return self.II if self.II > 0 else self.D


def Phi(z: float) -> float:
    return lib().orc_Phi(float(z))


def phi(z: float) -> float:
    return lib().orc_phi(float(z))


def F(family: int, z: float) -> float:
    """CDF of a family in z = (x - mu) / sigma, scale-matched to N(0, 1) (App. D)."""
    return lib().orc_F(int(family), float(z))


def f(family: int, z: float) -> float:
    """Density of a family in z = (x - mu) / sigma (App. D)."""
    return lib().orc_f(int(family), float(z))


def bin_masses(D: int, mu: float, sigma: float, family: int = GAUSSIAN) -> np.ndarray:
    """Eq. round over d = 0..D-1 with open boundary bins."""
    P = np.zeros(D, dtype=np.float64)
    lib().orc_bin_masses(C.c_int32(D), C.c_int32(family), C.c_double(mu), C.c_double(sigma), _p(P))
    return P


def asap_alap(op: OracleProblem):
    """Kahn order, ASAP, ALAP and critical path; rc 0 ok, 1 cycle, 2 horizon."""
    order = np.zeros(op.V, np.int32)
    asap = np.zeros(op.V, np.int32)
    alap = np.zeros(op.V, np.int32)
    cp = C.c_int32(0)
    rc = lib().orc_asap_alap(C.c_int32(op.V), C.c_int32(op.E), _p(op.src), _p(op.dst),
                             _p(op.lat), C.c_int32(op.D), _p(order), _p(asap), _p(alap),
                             C.byref(cp))
    return rc, order, asap, alap, cp.value


def hparams(tau=1e-2, rho=1e-4, alpha=1.0, w_res=1.0, w_mem=1.0, terms=DEP | COM | RES_OBJ,
            family=GAUSSIAN):
    return _Hparams(tau, rho, alpha, w_res, w_mem, terms, family)


def loss_grad(op: OracleProblem, hp, mu, sigma, lam):
    """Total loss of Sec. 3.3 and its gradient.  mu, sigma: (V, B); lam: (B, 3).

    Returns loss (B,), terms (B, 6), grad_mu (V, B), grad_sigma (V, B)."""
    mu = np.asarray(mu, np.float64)
    sigma = np.asarray(sigma, np.float64)
    V, B = mu.shape
    muT = np.ascontiguousarray(mu.T)
    sgT = np.ascontiguousarray(sigma.T)
    lam = np.ascontiguousarray(np.asarray(lam, np.float64).reshape(B, K))
    loss = np.zeros(B)
    terms = np.zeros((B, NT))
    gmu = np.zeros((B, V))
    gsg = np.zeros((B, V))
    lib().orc_loss_grad(C.byref(op.c), C.byref(hp), C.c_int32(B), _p(muT), _p(sgT), _p(lam),
                        _p(loss), _p(terms), _p(gmu), _p(gsg))
    return loss, terms, np.ascontiguousarray(gmu.T), np.ascontiguousarray(gsg.T)


def expected_hist(op: OracleProblem, mu, sigma, family: int = GAUSSIAN):
    """Expected usage U (C, Dh) and storage Reg (Dh,) of one restart."""
    mu = np.ascontiguousarray(np.asarray(mu, np.float64))
    sigma = np.ascontiguousarray(np.asarray(sigma, np.float64))
    U = np.zeros((op.C, op.Dh))
    R = np.zeros(op.Dh)
    lib().orc_expected_hist(C.byref(op.c), C.c_int32(family), _p(mu), _p(sigma), _p(U), _p(R))
    return U, R


def adam(theta, g, m, v, step, lr, beta1=0.9, beta2=0.999, eps=1e-8):
    """One in-place Adam step on float64 arrays (torch.optim.Adam semantics)."""
    for a in (theta, g, m, v):
        assert a.dtype == np.float64 and a.flags.c_contiguous
    lib().orc_adam(C.c_int64(theta.size), _p(theta), _p(g), _p(m), _p(v), C.c_int32(step),
                   C.c_double(lr), C.c_double(beta1), C.c_double(beta2), C.c_double(eps))


def round_half_up(mu) -> np.ndarray:
    mu = np.ascontiguousarray(np.asarray(mu, np.float64))
    s = np.zeros(mu.shape, np.int32)
    lib().orc_round(C.c_int64(mu.size), _p(mu), _p(s))
    return s


def legalize_regular(op: OracleProblem, order, asap, alap, s):
    """App. A Alg. 1 on one schedule s (V,), in the given topological order."""
    s = np.ascontiguousarray(np.asarray(s, np.int32)).copy()
    lib().orc_legalize_regular(C.byref(op.c), _p(np.ascontiguousarray(order, np.int32)),
                               _p(np.ascontiguousarray(asap, np.int32)),
                               _p(np.ascontiguousarray(alap, np.int32)), _p(s))
    return s


def legalize_modulo(op: OracleProblem, order, s):
    """App. A Alg. 2; returns (schedule, rc) with rc 1 when |V| sweeps did not settle."""
    s = np.ascontiguousarray(np.asarray(s, np.int32)).copy()
    rc = lib().orc_legalize_modulo(C.byref(op.c), _p(np.ascontiguousarray(order, np.int32)),
                                   _p(s))
    return s, rc


REPORT_FIELDS = ("n_dep_viol", "n_lat_viol", "n_rec_viol", "n_res_viol", "L_res", "L_com",
                 "L_mem", "L_mmem", "feasible", "res_ok")


def verify(op: OracleProblem, s) -> dict:
    """Sec. 2.1 discrete objectives and constraints of one schedule s (V,)."""
    s = np.ascontiguousarray(np.asarray(s, np.int32))
    r = _Report()
    lib().orc_verify(C.byref(op.c), _p(s), C.byref(r))
    out = {f: int(getattr(r, f)) for f in REPORT_FIELDS}
    out["peak"] = [int(r.peak[c]) for c in range(min(op.C, 16))]
    return out


def init_state(op: OracleProblem, B: int, kappa: float, sigma_min: float, mu0=None):
    """Sec. 3.3 Initialization for B restarts; kappa and sigma_min as the float32
    values the library receives.  Returns mu, sigma (V, B) float32."""
    rc, order, asap, alap, cp = asap_alap(op)
    assert rc == 0
    mu = np.zeros((B, op.V), np.float32)
    sg = np.zeros((B, op.V), np.float32)
    m0 = None if mu0 is None else np.ascontiguousarray(np.asarray(mu0, np.float32).T)
    for b in range(B):
        lib().orc_init_state(C.c_int32(op.V), _p(asap), _p(alap), C.c_double(float(np.float32(kappa))),
                             C.c_float(float(np.float32(sigma_min))), None if m0 is None else _p(m0[b]),
                             _p(mu[b]), _p(sg[b]))
    return np.ascontiguousarray(mu.T), np.ascontiguousarray(sg.T)


def outer_step(op: OracleProblem, terms: int, w_res: float, alpha: float, w_mem: float, it: int,
               s_legal, leg_ok, sigma_init, best: dict, state: dict):
    """One outer step of Alg. GauS on B restarts, in place on `best` (sched (V, B)
    int32, score (B,) float64, iter (B,) int32) and `state` (mu, sigma, m_mu, v_mu,
    m_sigma, v_sigma (V, B) float32, step (B,) int32).  s_legal (V, B): the
    legalization of round(mu); leg_ok (B,): its success.  The report of each
    legalized schedule is the oracle's own verify.  Returns moved (B,)."""
    rc, order, asap, alap, cp = asap_alap(op)
    V, B = np.asarray(s_legal).shape
    T = lambda a, dt: np.ascontiguousarray(np.asarray(a, dt).T)
    sl = T(s_legal, np.int32)
    si = T(sigma_init, np.float32)
    bs = T(best["sched"], np.int32)
    arr = {k: T(state[k], np.float32) for k in ("mu", "sigma", "m_mu", "v_mu", "m_sigma", "v_sigma")}
    score = np.ascontiguousarray(best["score"], np.float64).copy()
    biter = np.ascontiguousarray(best["iter"], np.int32).copy()
    step = np.ascontiguousarray(state["step"], np.int32).copy()
    moved = np.zeros(B, np.int32)
    for b in range(B):
        r = _Report()
        lib().orc_verify(C.byref(op.c), _p(sl[b]), C.byref(r))
        sc = np.zeros(1, np.float64); sc[0] = score[b]
        it_ = np.zeros(1, np.int32); it_[0] = biter[b]
        st_ = np.zeros(1, np.int32); st_[0] = step[b]
        moved[b] = lib().orc_outer_step(
            C.c_int32(V), C.c_int32(int(bool(leg_ok[b]))), _p(sl[b]), C.byref(r), C.c_uint32(terms),
            C.c_int32(op.II), C.c_double(float(np.float32(w_res))), C.c_double(float(np.float32(alpha))),
            C.c_double(float(np.float32(w_mem))), C.c_int32(it), _p(asap), _p(alap), _p(si[b]), _p(bs[b]),
            _p(sc), _p(it_), _p(arr["mu"][b]), _p(arr["sigma"][b]), _p(arr["m_mu"][b]), _p(arr["v_mu"][b]),
            _p(arr["m_sigma"][b]), _p(arr["v_sigma"][b]), _p(st_))
        score[b], biter[b], step[b] = sc[0], it_[0], st_[0]
    best["sched"][...] = bs.T
    best["score"][...] = score
    best["iter"][...] = biter
    for k, a in arr.items():
        state[k][...] = a.T
    state["step"][...] = step
    return moved
