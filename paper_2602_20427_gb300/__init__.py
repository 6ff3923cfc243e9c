"""GauS (arXiv 2602.20427) hot path on one GB300: thin Python binding of libgaus.so.

Argument marshalling only: every step of the path runs in the CUDA kernels of
``csrc/``.  Tensors are torch CUDA tensors in the (V, B) layout of
``include/gaus.h``; their ``data_ptr()`` and the current torch stream are
passed to the C ABI.  The library must be built (``build.build()``) and a CUDA
device present; there is no CPU fallback.
"""
from __future__ import annotations

import ctypes as C
import os
import re

import numpy as np

from .build import LIB as _LIB_PATH
from .build import build

__all__ = ["build", "lib", "Gaus", "default_hparams", "symbols_declared",
           "DEP", "COM", "RES_OBJ", "RES_VIOL", "REG_OBJ", "REC", "DEP_CF", "K", "NT", "STATUS",
           "GAUSSIAN", "LOGISTIC", "LAPLACE", "CAUCHY", "PEAK_FP32", "PEAK_EX2", "measure_peak",
           "PATH_AUTO", "PATH_FUSED", "PATH_MULTI"]

DEP, COM, RES_OBJ, RES_VIOL, REG_OBJ, REC = 1, 2, 4, 8, 16, 32
DEP_CF = 64  # continuous dependency penalty: a variant, not the paper's Eq. dep
K, NT = 3, 6
# CDF families (gaus_hparams.family): the normal, or in its place a scale-matched
# logistic, Laplace or Cauchy CDF (App. D)
GAUSSIAN, LOGISTIC, LAPLACE, CAUCHY = 0, 1, 2, 3
STATUS = {0: "OK", 1: "EINVAL", 2: "ECYCLE", 3: "EHORIZON", 4: "ENOMEM", 5: "ECUDA",
          6: "ENONFINITE", 7: "ENOTCONV", 8: "ETIMEOUT"}

_HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "gaus.h")


class GausError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{STATUS.get(code, code)}: {msg}")
        self.code = code


class Problem(C.Structure):
    _fields_ = [("V", C.c_int32), ("E", C.c_int32),
                ("succ_ptr", C.c_void_p), ("succ_idx", C.c_void_p),
                ("pred_ptr", C.c_void_p), ("pred_idx", C.c_void_p),
                ("latency", C.c_void_p), ("res_class", C.c_void_p), ("C", C.c_int32),
                ("limit", C.c_void_p), ("demand", C.c_void_p), ("bits", C.c_void_p),
                ("n_back", C.c_int32), ("back_src", C.c_void_p), ("back_dst", C.c_void_p),
                ("back_dist", C.c_void_p), ("D", C.c_int32), ("II", C.c_int32), ("B", C.c_int32)]


class Hparams(C.Structure):
    _fields_ = [(n, C.c_float) for n in ("tau", "rho", "lambda0", "alpha", "w_res", "w_mem", "lr",
                                         "beta1", "beta2", "eps", "window_k", "sigma_min")] + \
               [("terms", C.c_uint32), ("family", C.c_int32)]


class Report(C.Structure):
    _fields_ = [("n_dep_viol", C.c_int64), ("n_lat_viol", C.c_int64), ("n_rec_viol", C.c_int64),
                ("n_res_viol", C.c_int64), ("L_res", C.c_int64), ("L_com", C.c_int64),
                ("L_mem", C.c_int64), ("L_mmem", C.c_int64), ("peak", C.c_int64 * 16),
                ("feasible", C.c_int32), ("res_ok", C.c_int32)]


class Best(C.Structure):
    _fields_ = [("sched", C.c_void_p), ("score", C.c_void_p), ("iter", C.c_void_p)]


class State(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("mu", "sigma", "m_mu", "v_mu", "m_sigma", "v_sigma",
                                          "lambda_", "step", "loss", "terms", "status")]


REPORT_FIELDS = ("n_dep_viol", "n_lat_viol", "n_rec_viol", "n_res_viol", "L_res", "L_com",
                 "L_mem", "L_mmem", "feasible", "res_ok")

_lib = None


def symbols_declared() -> list[str]:
    """Entry points declared in include/gaus.h."""
    txt = open(_HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:gaus_status|void|const char \*)\s*(gaus_\w+)\s*\(", txt, re.M)))


def lib():
    """Load libgaus.so; raises if it was not built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: run __graft_entry__.build() first")
        L = C.CDLL(_LIB_PATH)
        for name in symbols_declared():
            getattr(L, name)
        L.gaus_last_error.restype = C.c_char_p
        L.gaus_last_error.argtypes = [C.c_void_p]
        L.gaus_destroy.restype = None
        L.gaus_destroy.argtypes = [C.c_void_p]
        for name in symbols_declared():
            if name not in ("gaus_last_error", "gaus_destroy"):
                getattr(L, name).restype = C.c_int
        _lib = L
    return _lib


PEAK_FP32, PEAK_EX2 = 0, 1
PATH_AUTO, PATH_FUSED, PATH_MULTI = 0, 1, 2


def measure_peak(what: int, stream=None) -> float:
    """gaus_measure_peak: FP32 FMA FLOP/s (PEAK_FP32) or SFU exp2 results/s (PEAK_EX2)
    of the current device, from the library's microbenchmark."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    v = C.c_double()
    rc = lib().gaus_measure_peak(C.c_int32(what), C.byref(v), C.c_void_p(s.cuda_stream))
    if rc != 0:
        raise GausError(rc, "gaus_measure_peak failed")
    return v.value


def default_hparams(**kw) -> Hparams:
    h = Hparams()
    rc = lib().gaus_default_hparams(C.byref(h))
    assert rc == 0
    for k, v in kw.items():
        setattr(h, k, v)
    return h


def _csr(V, key, val):
    order = np.lexsort((val, key))
    ptr = np.zeros(V + 1, np.int32)
    np.add.at(ptr, key + 1, 1)
    return np.cumsum(ptr).astype(np.int32), np.ascontiguousarray(val[order].astype(np.int32))


class Gaus:
    """One GauS problem on the current CUDA device (gaus_create ... gaus_destroy)."""

    def __init__(self, prob, B: int, hparams: Hparams | None = None, stream=None):
        import torch
        self.torch = torch
        self.V, self.D, self.II, self.C, self.B = int(prob.V), int(prob.D), int(prob.II), int(prob.C), int(B)
        src = np.asarray(prob.src, np.int64)
        dst = np.asarray(prob.dst, np.int64)
        self._keep = []

        def arr(x, dt):
            a = np.ascontiguousarray(np.asarray(x, dt))
            self._keep.append(a)
            return a.ctypes.data if a.size else None

        sp, si = _csr(self.V, src, dst)
        pp, pi = _csr(self.V, dst, src)
        nb = int(np.asarray(prob.bsrc).size)
        self._p = Problem(self.V, int(src.size), arr(sp, np.int32), arr(si, np.int32), arr(pp, np.int32),
                          arr(pi, np.int32), arr(prob.lat, np.int32), arr(prob.cls, np.int32), self.C,
                          arr(prob.limit, np.float32), arr(prob.demand, np.int32), arr(prob.bits, np.int32),
                          nb, arr(prob.bsrc, np.int32), arr(prob.bdst, np.int32), arr(prob.bdist, np.int32),
                          self.D, self.II, self.B)
        self.hp = hparams if hparams is not None else default_hparams()
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        ctx = C.c_void_p()
        rc = lib().gaus_create(C.byref(self._p), C.byref(self.hp), C.c_void_p(self.stream.cuda_stream),
                               C.byref(ctx))
        if rc != 0:
            raise GausError(rc, lib().gaus_last_error(None).decode())
        self._ctx = ctx

    # -- helpers
    def _check(self, rc):
        if rc != 0:
            raise GausError(rc, lib().gaus_last_error(self._ctx).decode())

    def _dev(self, t, dtype, shape):
        torch = self.torch
        assert t.is_cuda and t.dtype == dtype and t.is_contiguous() and tuple(t.shape) == tuple(shape), \
            (t.device, t.dtype, t.shape, shape)
        return C.c_void_p(t.data_ptr())

    def close(self):
        if getattr(self, "_ctx", None):
            lib().gaus_destroy(self._ctx)
            self._ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_hparams(self, hp: Hparams):
        self._check(lib().gaus_set_hparams(self._ctx, C.byref(hp)))
        self.hp = hp

    def bounds(self):
        asap = np.zeros(self.V, np.int32)
        alap = np.zeros(self.V, np.int32)
        cp = C.c_int32()
        self._check(lib().gaus_bounds(self._ctx, C.c_void_p(asap.ctypes.data), C.c_void_p(alap.ctypes.data),
                                      C.byref(cp)))
        return asap, alap, cp.value

    PLAN_KEYS = ("fused", "fused_launches_per_call", "launches_per_iteration", "restart_groups",
                 "blocks_per_group", "restarts_per_group", "table_row_points", "fused_smem_bytes", "sms",
                 "node_segments", "edge_chunks", "fused_threads", "path_mode", "fused_calls", "multi_iterations",
                 "path_choices")

    def set_path(self, mode):
        """gaus_set_path: PATH_AUTO (choose per call), PATH_FUSED or PATH_MULTI."""
        self._check(lib().gaus_set_path(self._ctx, C.c_int32(mode)))

    def plan_info(self):
        """The execution plan for the current sizes and hyperparameters (gaus_plan_info)."""
        out = (C.c_int64 * len(self.PLAN_KEYS))()
        self._check(lib().gaus_plan_info(self._ctx, out, C.c_int32(len(self.PLAN_KEYS))))
        return dict(zip(self.PLAN_KEYS, [int(x) for x in out]))

    def check_barrier_timeout(self, state, limit_ns):
        """gaus_check_barrier_timeout: one fused iteration whose barriers never complete."""
        self._check(lib().gaus_check_barrier_timeout(self._ctx, C.byref(self._state(state)), C.c_uint64(limit_ns)))

    # -- entry points
    def loss_grad(self, mu, sigma, lam, out=None):
        torch = self.torch
        VB, f32 = (self.V, self.B), torch.float32
        if out is None:
            out = dict(grad_mu=torch.empty(VB, dtype=f32, device=mu.device),
                       grad_sigma=torch.empty(VB, dtype=f32, device=mu.device),
                       loss=torch.empty(self.B, dtype=f32, device=mu.device),
                       terms=torch.empty((self.B, NT), dtype=f32, device=mu.device),
                       status=torch.empty(self.B, dtype=torch.int32, device=mu.device))
        self._check(lib().gaus_loss_grad(
            self._ctx, self._dev(mu, f32, VB), self._dev(sigma, f32, VB), self._dev(lam, f32, (self.B, K)),
            self._dev(out["grad_mu"], f32, VB), self._dev(out["grad_sigma"], f32, VB),
            self._dev(out["loss"], f32, (self.B,)), self._dev(out["terms"], f32, (self.B, NT)),
            self._dev(out["status"], torch.int32, (self.B,))))
        return out

    def adam_step(self, mu, sigma, grad_mu, grad_sigma, m_mu, v_mu, m_sigma, v_sigma, lam, terms, step):
        torch = self.torch
        VB, f32 = (self.V, self.B), torch.float32
        self._check(lib().gaus_adam_step(
            self._ctx, self._dev(mu, f32, VB), self._dev(sigma, f32, VB), self._dev(grad_mu, f32, VB),
            self._dev(grad_sigma, f32, VB), self._dev(m_mu, f32, VB), self._dev(v_mu, f32, VB),
            self._dev(m_sigma, f32, VB), self._dev(v_sigma, f32, VB), self._dev(lam, f32, (self.B, K)),
            self._dev(terms, f32, (self.B, NT)), C.c_int32(step)))

    def new_state(self, mu, sigma, lambda0=None):
        """Device state for iterate(): copies of mu/sigma, zero moments, lambda = lambda0."""
        torch = self.torch
        dev = mu.device
        lam0 = float(self.hp.lambda0 if lambda0 is None else lambda0)
        z = lambda: torch.zeros((self.V, self.B), dtype=torch.float32, device=dev)
        return dict(mu=mu.clone(), sigma=sigma.clone(), m_mu=z(), v_mu=z(), m_sigma=z(), v_sigma=z(),
                    lambda_=torch.full((self.B, K), lam0, dtype=torch.float32, device=dev),
                    step=torch.zeros(self.B, dtype=torch.int32, device=dev),
                    loss=torch.zeros(self.B, dtype=torch.float32, device=dev),
                    terms=torch.zeros((self.B, NT), dtype=torch.float32, device=dev),
                    status=torch.zeros(self.B, dtype=torch.int32, device=dev))

    def iterate(self, n, state):
        """n fused iterations (gaus_iterate) on the state dict of new_state()/init_state()."""
        self._check(lib().gaus_iterate(self._ctx, C.c_int32(n), C.byref(self._state(state))))

    def profile_iterate(self, n, state):
        """Mean per-iteration durations (ms) over n iterations launched kernel by kernel:
        [node pass, edge pass, reductions + finalize, update] (gaus_profile_iterate)."""
        ms = (C.c_double * 4)(0.0, 0.0, 0.0, 0.0)
        self._check(lib().gaus_profile_iterate(self._ctx, C.c_int32(n), C.byref(self._state(state)), ms))
        return list(ms)

    PHASE_KEYS = ("p1_crit", "p2_crit", "p3_crit", "p1_mean", "p2_mean", "p3_mean", "bar1", "bar2",
                  "iteration", "p1_max", "p2_max", "p3_max")

    def profile_phases(self, n, state):
        """Phase profile of n fused iterations of the persistent kernel (ms, means over
        the iterations; gaus_profile_phases): critical path, mean and slowest block of
        each phase, the two barrier latencies and the iteration time."""
        out = (C.c_double * 12)()
        self._check(lib().gaus_profile_phases(self._ctx, C.c_int32(n), C.byref(self._state(state)), out))
        return dict(zip(self.PHASE_KEYS, list(out)))

    def _state(self, state):
        torch = self.torch
        VB, f32 = (self.V, self.B), torch.float32
        return State(*(self._dev(state[k], f32, VB).value for k in ("mu", "sigma", "m_mu", "v_mu", "m_sigma",
                                                                     "v_sigma")),
                     self._dev(state["lambda_"], f32, (self.B, K)).value,
                     self._dev(state["step"], torch.int32, (self.B,)).value,
                     self._dev(state["loss"], f32, (self.B,)).value,
                     self._dev(state["terms"], f32, (self.B, NT)).value,
                     self._dev(state["status"], torch.int32, (self.B,)).value)

    def _best(self, best):
        torch = self.torch
        return Best(self._dev(best["sched"], torch.int32, (self.V, self.B)).value,
                    self._dev(best["score"], torch.float64, (self.B,)).value,
                    self._dev(best["iter"], torch.int32, (self.B,)).value)

    def init_state(self, kappa=1.0 / 6.0, mu0=None, device="cuda", out=None):
        """Alg. GauS initialization (gaus_init_state): a fresh state (mu = mu0 or the
        ASAP/ALAP midpoint, sigma = max(kappa (ALAP - ASAP), sigma_min)), the
        sigma a reset returns to, and an empty best.  out = (state, sigma_init,
        best) re-initialises those buffers in place."""
        torch = self.torch
        VB = (self.V, self.B)
        if out is not None:
            state, sigma_init, best = out
            s, bst = self._state(state), self._best(best)
            m0 = None if mu0 is None else self._dev(mu0, torch.float32, VB)
            self._check(lib().gaus_init_state(self._ctx, m0, C.c_float(kappa), C.byref(s),
                                              self._dev(sigma_init, torch.float32, VB), C.byref(bst)))
            return out
        z = lambda: torch.empty(VB, dtype=torch.float32, device=device)
        state = dict(mu=z(), sigma=z(), m_mu=z(), v_mu=z(), m_sigma=z(), v_sigma=z(),
                     lambda_=torch.empty((self.B, K), dtype=torch.float32, device=device),
                     step=torch.empty(self.B, dtype=torch.int32, device=device),
                     loss=torch.zeros(self.B, dtype=torch.float32, device=device),
                     terms=torch.zeros((self.B, NT), dtype=torch.float32, device=device),
                     status=torch.empty(self.B, dtype=torch.int32, device=device))
        sigma_init = z()
        best = dict(sched=torch.zeros(VB, dtype=torch.int32, device=device),
                    score=torch.empty(self.B, dtype=torch.float64, device=device),
                    iter=torch.empty(self.B, dtype=torch.int32, device=device))
        s, bst = self._state(state), self._best(best)
        m0 = None if mu0 is None else self._dev(mu0, torch.float32, VB)
        self._check(lib().gaus_init_state(self._ctx, m0, C.c_float(kappa), C.byref(s),
                                          self._dev(sigma_init, torch.float32, VB), C.byref(bst)))
        return state, sigma_init, best

    def outer_step(self, state, sched, leg_status, rep, it, sigma_init, best, moved=None):
        """One outer step (gaus_outer_step); returns the nodes legalization moved per restart."""
        torch = self.torch
        if moved is None:
            moved = torch.empty(self.B, dtype=torch.int32, device=sched.device)
        s, bst = self._state(state), self._best(best)
        self._check(lib().gaus_outer_step(self._ctx, self._dev(sched, torch.int32, (self.V, self.B)),
                                          self._dev(leg_status, torch.int32, (self.B,)),
                                          C.c_void_p(rep.data_ptr()), C.c_int32(it),
                                          self._dev(sigma_init, torch.float32, (self.V, self.B)), C.byref(s),
                                          C.byref(bst), self._dev(moved, torch.int32, (self.B,))))
        return moved

    def solve(self, n_periods, period, state, sigma_init, best, iter0=0, work=None):
        """n_periods periods of Alg. GauS on the device (gaus_solve); returns the work
        buffers (last legalized schedules, their status and reports, nodes moved)."""
        torch = self.torch
        dev = state["mu"].device
        if work is None:
            work = dict(sched=torch.empty((self.V, self.B), dtype=torch.int32, device=dev),
                        leg_status=torch.empty(self.B, dtype=torch.int32, device=dev),
                        rep=torch.empty(C.sizeof(Report) * self.B, dtype=torch.uint8, device=dev),
                        moved=torch.empty(self.B, dtype=torch.int32, device=dev))
        s, bst = self._state(state), self._best(best)
        self._check(lib().gaus_solve(self._ctx, C.c_int32(n_periods), C.c_int32(period), C.c_int32(iter0),
                                     C.byref(s), self._dev(sigma_init, torch.float32, (self.V, self.B)),
                                     C.byref(bst), self._dev(work["sched"], torch.int32, (self.V, self.B)),
                                     self._dev(work["leg_status"], torch.int32, (self.B,)),
                                     C.c_void_p(work["rep"].data_ptr()),
                                     self._dev(work["moved"], torch.int32, (self.B,))))
        return work

    def round(self, mu, sched=None):
        torch = self.torch
        if sched is None:
            sched = torch.empty((self.V, self.B), dtype=torch.int32, device=mu.device)
        self._check(lib().gaus_round(self._ctx, self._dev(mu, torch.float32, (self.V, self.B)),
                                     self._dev(sched, torch.int32, (self.V, self.B))))
        return sched

    def legalize(self, mu, sched=None, status=None):
        torch = self.torch
        if sched is None:
            sched = torch.empty((self.V, self.B), dtype=torch.int32, device=mu.device)
        if status is None:
            status = torch.empty(self.B, dtype=torch.int32, device=mu.device)
        self._check(lib().gaus_legalize(self._ctx, self._dev(mu, torch.float32, (self.V, self.B)),
                                        self._dev(sched, torch.int32, (self.V, self.B)),
                                        self._dev(status, torch.int32, (self.B,))))
        return sched, status

    def verify_raw(self, sched, rep=None):
        """Reports as a device byte tensor (B * sizeof(gaus_report))."""
        torch = self.torch
        n = C.sizeof(Report) * self.B
        if rep is None:
            rep = torch.empty(n, dtype=torch.uint8, device=sched.device)
        self._check(lib().gaus_verify(self._ctx, self._dev(sched, torch.int32, (self.V, self.B)),
                                      C.c_void_p(rep.data_ptr())))
        return rep

    def verify(self, sched):
        """List of B report dicts (copied to the host)."""
        raw = self.verify_raw(sched).cpu().numpy().tobytes()
        out = []
        for b in range(self.B):
            r = Report.from_buffer_copy(raw[b * C.sizeof(Report):(b + 1) * C.sizeof(Report)])
            d = {f: int(getattr(r, f)) for f in REPORT_FIELDS}
            d["peak"] = [int(r.peak[c]) for c in range(min(self.C, 16))]
            out.append(d)
        return out
