#!/usr/bin/env python
"""GauS hot-path benchmark: fused loss + gradient + Adam iterations/s x B restarts.

One step = one complete batched solve of Alg. GauS on the logic-network
workload (V = 10,000, B = 64 restarts) from its seeded initial state: the state
is initialised (means and deviations copied in, Adam moments and step zeroed,
multipliers set to lambda_0), then `--iters` fused iterations (gaus_iterate:
loss, gradient, Adam, multiplier update; Sec. 3.3) run, with a round + legalize
(App. A) and a verify (Sec. 2.1) of all B restarts every `--period` iterations.
Every step does the same work, so the number does not depend on --steps.

Prints one JSON line.  `--impl reference` times the fp64 CPU oracle on the same
workload and metric (bounded sample per step).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "loss+grad+Adam iterations/s x B restarts (logic-network DAG, |V|=10k)"
UNIT = "restart-iterations/s"
FP32_LANES_PER_SM = 128
SM_COUNT = 152
SM_MAX_MHZ = 2070.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--iters", type=int, default=2000, help="fused iterations per solve (one step)")
    ap.add_argument("--period", type=int, default=100, help="iterations between legalize + verify")
    ap.add_argument("--impl", default="gaus", choices=["gaus", "reference"])
    ap.add_argument("--phase-probe", type=int, default=None, metavar="N",
                    help="run N iterations kernel by kernel, then one more, print the phase times and exit "
                         "(a fixed launch sequence for ncu captures at iteration N)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-solver", action="store_true", help="skip the complete-solver runs (gaus_solve)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-families", action="store_true", help="skip the CDF-family timings")
    ap.add_argument("--restarts", type=int, default=64,
                    help="restarts per rank (64 is the benchmark configuration; others for scaling studies)")
    ap.add_argument("--profile-range", action="store_true",
                    help="bracket the timed steps with cudaProfilerStart/Stop (for ncu --profile-from-start off)")
    return ap.parse_args()


def workload(rank=0, B=64):
    """The benchmark workload of one rank: the same logic-network DAG on every rank,
    and B (64) restarts of its own (initial state seeded by the rank), so the ranks'
    restarts are independent and need no data-path collective (weak scaling)."""
    p = W.logic_network(1)
    mu, sg = W.init_state(p, B, seed=1 + rank)
    return p, B, mu, sg


def max_over_ranks(ms, world, dist=None, device="cpu"):
    """The job's time: the slowest rank's (max all-reduce; the only collective)."""
    if world <= 1:
        return float(ms)
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(steps, iters, B, world, ms):
    """Whole-job restart-iterations/s: every rank's units over the slowest rank's time."""
    return steps * iters * B * world / (ms / 1e3)


def describe(p, B, iters, period=None):
    return {"workload": f"{p.name}: AND/INV logic network, V={p.V}, E={p.E}, depth 120, "
                        f"D={p.D}, 2 classes (AND limit 64, INV unlimited), unit latency, "
                        f"Formulation A terms (Res LSE + ReLU, Com, Dep)",
            "B": B, "V": p.V, "E": p.E, "D": p.D, "iterations_per_step": iters,
            "legalize_verify_every": period,
            "init": "mu = ASAP + N(0, 2), sigma = 1.5 (seeded)", "tau": 1e-2, "rho": 1e-4, "lr": 1e-2,
            "window_k": 6.0}


# ----------------------------------------------------------------- clocks
class ClockSampler:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.rows = []
        self.proc = None

    def start(self):
        try:
            cmd = ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.gpu_id is not None:
                cmd += ["-i", str(self.gpu_id)]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                self.rows.append(parts)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in self.rows if r[2].replace(".", "").isdigit()]
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in self.rows:
            for name, val in zip(names, r[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(self.rows)}


# ----------------------------------------------------------------- algorithmic work
def algorithmic_flops(torch, mu, sg, src, dst, k, D):
    """FP32 work of one node/edge pass under the cost model of the design notes:
    20 flop per CDF point and 8 flop per edge-bin, with the points of each
    (node, restart) window of +-k sigma (bins = points + 1)."""
    a = torch.clamp(torch.ceil(mu - k * sg - 0.5), 0, D - 1)
    b = torch.clamp(torch.floor(mu + k * sg - 0.5), -1, D - 2)
    bins = (b - a + 2).to(torch.float64)                  # (V, B)
    n_pt = float(bins.sum())
    # dependency edge: producer bins; communication: producer + consumer bins
    n_eb = float((2.0 * bins[src] + bins[dst]).sum())
    return 20.0 * n_pt + 8.0 * n_eb, n_pt, n_eb


def measured_hbm_gbs():
    """HBM copy bandwidth from MEASURED_PEAKS.json, else the fallback of an earlier GB300 measurement."""
    try:
        return float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))["hbm_gbs"])
    except (OSError, KeyError, ValueError):
        return 6800.0


def profiled_traffic():
    """DRAM bytes per k_edges launch from the committed ncu summary, or None when the
    kernel sources changed since that capture."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", "k_edges_logic_network_v10000_b64.md")
    if not os.path.exists(prof):
        return None
    txt = open(prof).read()
    want = {}
    for line in txt.splitlines():
        if ":" in line and line.split(":")[0] in ("dram-bytes-per-launch", "source-sha256"):
            want[line.split(":")[0]] = line.split(":", 1)[1].strip()
    lines = []
    for f in ("gaus_kernels.cuh", "gaus_device.cuh"):
        path = os.path.join(ROOT, "paper_2602_20427_gb300", "csrc", f)
        h = hashlib.sha256(open(path, "rb").read()).hexdigest()
        lines.append(f"{h}  paper_2602_20427_gb300/csrc/{f}\n")
    cur = hashlib.sha256("".join(lines).encode()).hexdigest()
    if want.get("source-sha256") != cur or "dram-bytes-per-launch" not in want:
        return None
    return float(want["dram-bytes-per-launch"])


def gpu_arm(args):
    import torch
    import torch.distributed as dist

    import paper_2602_20427_gb300 as g

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    g.build()
    p, B, mu0, sg0 = workload(rank, args.restarts)
    hp = g.default_hparams(terms=p.terms)
    ctx = g.Gaus(p, B, hp)
    iters, period = args.iters, args.period
    assert iters % period == 0, "--iters must be a multiple of --period"
    dmu0, dsg0 = torch.from_numpy(mu0).cuda(), torch.from_numpy(sg0).cuda()
    st = ctx.new_state(dmu0, dsg0, hp.lambda0)
    sched = torch.empty((p.V, B), dtype=torch.int32, device="cuda")
    lstat = torch.empty(B, dtype=torch.int32, device="cuda")
    rep = torch.empty(B * 200, dtype=torch.uint8, device="cuda")
    reg = bool(p.terms & W.REG_OBJ)
    # per iteration: k_nodes, k_edges, k_reduce, k_finalize, k_update [+ k_reg_fwd, k_reduce_reg,
    # k_reg_bwd]; per period: the legalization kernel and the verifier's two passes
    launches_per_iter = 5 + (3 if reg else 0)
    launches_per_step = iters * launches_per_iter + (iters // period) * 3

    def init_state(mu_src, sg_src):
        st["mu"].copy_(mu_src, non_blocking=True)
        st["sigma"].copy_(sg_src, non_blocking=True)
        for kk in ("m_mu", "v_mu", "m_sigma", "v_sigma", "loss", "terms"):
            st[kk].zero_()
        st["step"].zero_()
        st["status"].zero_()
        st["lambda_"].fill_(hp.lambda0)

    def solve():
        for _ in range(iters // period):
            ctx.iterate(period, st)
            ctx.legalize(st["mu"], sched, lstat)
            ctx.verify_raw(sched, rep)

    def step():
        init_state(dmu0, dsg0)
        solve()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device="cuda")
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(local).uuid)
    except Exception:
        gpu_id = None
    # this device's FP32 FMA and SFU exp2 throughput (the library's microbenchmark)
    fp32_peak = g.measure_peak(g.PEAK_FP32)
    ex2_peak = g.measure_peak(g.PEAK_EX2)
    hbm_peak = measured_hbm_gbs() * 1e9
    sampler = ClockSampler(gpu_id) if rank == 0 else None
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
        time.sleep(0.5)
    wall0 = time.perf_counter()
    if args.profile_range:
        torch.cuda.profiler.start()              # ncu --profile-from-start off: the timed steps only
    for k in range(args.steps):
        flush.fill_(k & 255)                     # L2 flush between steps (outside the events)
        evs[k][0].record()
        step()
        evs[k][1].record()
    torch.cuda.synchronize()
    if args.profile_range:
        torch.cuda.profiler.stop()
    wall = time.perf_counter() - wall0
    clocks = sampler.stop() if sampler else None
    step_ms = [a.elapsed_time(b) for a, b in evs]
    ms = sum(step_ms)
    if world > 1:
        dist.barrier()
    ms = max_over_ranks(ms, world, dist, "cuda")
    status_ok = bool(int(st["status"].abs().sum()) == 0)
    feasible = int((lstat == 0).sum())
    units = args.steps * iters * B * world
    value = job_throughput(args.steps, iters, B, world, ms)

    # ---- legalize + verify alone (part of every step above; reported separately)
    lv = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    lv[0].record()
    for _ in range(10):
        ctx.legalize(st["mu"], sched, lstat)
        ctx.verify_raw(sched, rep)
    lv[1].record()
    torch.cuda.synchronize()
    legalize_verify_ms = lv[0].elapsed_time(lv[1]) / 10

    # ---- phase timing and algorithmic work along one solve (no graph, events between phases)
    init_state(dmu0, dsg0)
    src = torch.from_numpy(np.asarray(p.src, np.int64)).cuda()
    dst = torch.from_numpy(np.asarray(p.dst, np.int64)).cuda()
    ph_ms = np.zeros(4)
    t_edges_total, t_nodes_total, npt_total, neb_total = 0.0, 0.0, 0.0, 0.0
    t_star, t_star_by = 0.0, {"hbm": 0, "sfu": 0, "fp32": 0}
    state_bytes = 48.0 * p.V * B + (2.0 * p.E + 6.0 * p.V) * 4.0   # per iteration, design-independent
    fwd_first = fwd_last = None
    nchunk = iters // period
    for k in range(nchunk):
        _, n0, e0 = algorithmic_flops(torch, st["mu"], st["sigma"], src, dst, hp.window_k, p.D)
        kms = np.array(ctx.profile_iterate(period, st))
        _, n1, e1 = algorithmic_flops(torch, st["mu"], st["sigma"], src, dst, hp.window_k, p.D)
        ph_ms += kms / nchunk
        npt_total += period * 0.5 * (n0 + n1)
        neb_total += period * 0.5 * (e0 + e1)
        pts, ebs = 0.5 * (n0 + n1), 0.5 * (e0 + e1)
        bound = {"hbm": state_bytes / hbm_peak, "sfu": pts / ex2_peak, "fp32": (20.0 * pts + 8.0 * ebs) / fp32_peak}
        t_star += period * max(bound.values())
        t_star_by[max(bound, key=bound.get)] += period
        t_nodes_total += period * kms[0] * 1e-3
        t_edges_total += period * kms[1] * 1e-3
        fwd_first = kms[1] if fwd_first is None else fwd_first
        fwd_last = kms[1]
    achieved = 8.0 * neb_total / t_edges_total / 1e12           # edge pass: 8 flop per edge-bin
    nodes_achieved = 20.0 * npt_total / t_nodes_total / 1e12    # node pass: 20 flop per CDF point
    peak = SM_COUNT * FP32_LANES_PER_SM * 2 * SM_MAX_MHZ * 1e6 / 1e12
    traffic = profiled_traffic()

    # ---- steady state at fixed sigma: the initial state with lr = 1e-20 (an Adam step is
    # at most ~lr, far below one ulp of mu or sigma, so the windows never shrink)
    hp0 = g.default_hparams(terms=p.terms, lr=1e-20)
    ctx0 = g.Gaus(p, B, hp0)
    st0 = ctx0.new_state(dmu0, dsg0, hp0.lambda0)
    ctx0.iterate(20, st0)
    ev0 = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    n_fixed = 200
    torch.cuda.synchronize()
    ev0[0].record()
    ctx0.iterate(n_fixed, st0)
    ev0[1].record()
    torch.cuda.synchronize()
    fixed_ms = ev0[0].elapsed_time(ev0[1]) / n_fixed
    fixed_ph = ctx0.profile_iterate(20, st0)
    ctx0.close()
    steady = {"value": B / (fixed_ms / 1e3), "unit": UNIT, "sigma": 1.5, "ms_per_iteration": fixed_ms,
              "k_edges_ms": fixed_ph[1],
              "note": "initial state of the same workload with lr = 1e-20, so every iteration has the "
                      "initial +-6 sigma windows (the most expensive point of the run)"}

    # ---- the complete solver: the outer loop of Alg. GauS on the device (gaus_solve)
    # from the kappa initialization, one solve of the same length; anytime quality
    solver = None
    if not args.no_solver:
        ctxS = g.Gaus(p, B, hp)
        bufs = ctxS.init_state(kappa=1.0 / 6.0)
        work = ctxS.solve(1, period, *bufs)                    # captures the graphs
        ctxS.init_state(kappa=1.0 / 6.0, out=bufs)
        evS = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        torch.cuda.synchronize()
        evS[0].record()
        ctxS.solve(iters // period, period, *bufs, work=work)
        evS[1].record()
        torch.cuda.synchronize()
        sms = evS[0].elapsed_time(evS[1])
        bsc = bufs[2]["score"].cpu().numpy()
        found = np.isfinite(bsc)
        solver = {"value": iters * B / (sms / 1e3), "unit": UNIT, "ms": sms,
                  "init": "kappa = 1/6: sigma = max(kappa (ALAP - ASAP), sigma_min), mu = (ASAP + ALAP) / 2",
                  "periods": iters // period, "period": period,
                  "restarts_with_feasible_best": int(found.sum()),
                  "best_score_min": float(bsc[found].min()) if found.any() else None,
                  "best_score_mean": float(bsc[found].mean()) if found.any() else None,
                  "score": "L_res + alpha L_com of the best legal schedule (no resource overflow)"}
        # the same solver from the timed workload's initialization (mu = ASAP + N(0, 2),
        # sigma = 1.5), twice as long: how many restarts reach a feasible schedule, and when
        bufs = ctxS.init_state(kappa=1.0 / 6.0, mu0=dmu0, out=bufs)
        bufs[0]["sigma"].copy_(dsg0)
        bufs[1].copy_(dsg0)
        n_long = 2 * iters // period
        torch.cuda.synchronize()
        evS[0].record()
        ctxS.solve(n_long, period, *bufs, work=work)
        evS[1].record()
        torch.cuda.synchronize()
        lms = evS[0].elapsed_time(evS[1])
        bsc = bufs[2]["score"].cpu().numpy()
        bit = bufs[2]["iter"].cpu().numpy()
        found = np.isfinite(bsc)
        solver["from_workload_init"] = {
            "iterations": n_long * period, "restart_iterations_per_s": n_long * period * B / (lms / 1e3),
            "restarts_with_feasible_best": int(found.sum()),
            "best_found_at_iteration_min": int(bit[found].min()) if found.any() else None,
            "best_found_at_iteration_median": float(np.median(bit[found])) if found.any() else None,
            "best_score_min": float(bsc[found].min()) if found.any() else None,
            "best_score_mean": float(bsc[found].mean()) if found.any() else None}
        ctxS.close()

    # ---- Formulation C (modulo scheduling) sweep: II in {MII, 1.25 MII, 1.5 MII} on the
    # loop-body workload, the complete solver from that workload's initialization
    # (mu = ASAP + N(0, 2), sigma = 1.5; the kappa initialization spans the whole
    # horizon here, D = 3 II)
    sweep = None
    if not args.no_solver and rank == 0:
        sweep = []
        for factor in (1.0, 1.25, 1.5):
            pm = W.modulo_loop(1, ii_factor=factor)
            Bm = 32
            mu_m, sg_m = W.init_state(pm, Bm, seed=1)
            mu_m = torch.from_numpy(mu_m).cuda()
            hpm = g.default_hparams(terms=pm.terms)
            cm = g.Gaus(pm, Bm, hpm)

            def init_m(out=None):
                bufs_m = cm.init_state(kappa=1.0 / 6.0, mu0=mu_m, out=out)
                bufs_m[0]["sigma"].fill_(float(sg_m[0, 0]))
                bufs_m[1].fill_(float(sg_m[0, 0]))
                return bufs_m

            bm = init_m()
            wm = cm.solve(1, period, *bm)
            init_m(out=bm)
            evm = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            n_per = 10
            torch.cuda.synchronize()
            evm[0].record()
            cm.solve(n_per, period, *bm, work=wm)
            evm[1].record()
            torch.cuda.synchronize()
            mms = evm[0].elapsed_time(evm[1])
            sc = bm[2]["score"].cpu().numpy()
            fnd = np.isfinite(sc)
            ls = wm["leg_status"].cpu().numpy()
            sweep.append({"ii_factor": factor, "II": pm.II, "D": pm.D, "V": pm.V, "E": pm.E, "back_edges": pm.NB,
                          "B": Bm, "iterations": n_per * period,
                          "restart_iterations_per_s": n_per * period * Bm / (mms / 1e3),
                          "restarts_with_feasible_best": int(fnd.sum()),
                          "best_score_min": float(sc[fnd].min()) if fnd.any() else None,
                          "best_score_mean": float(sc[fnd].mean()) if fnd.any() else None,
                          "last_legalize_not_converged": int((ls == 7).sum()),
                          "init": "mu = ASAP + N(0, 2), sigma = 1.5 (seeded)",
                          "score": "w_mem L_mmem of the best legal schedule (no resource overflow)"})
            cm.close()

    # ---- CDF families (App. D): the first 100 fused iterations of the same workload
    # from the same initialization with the normal, logistic, Laplace and Cauchy
    # relaxations (heavier tails: wider windows), and the normal with the continuous
    # dependency penalty in place of the binned Eq. dep
    families = None
    if not args.no_families and rank == 0:
        families = []
        cf_terms = (p.terms & ~g.DEP) | g.DEP_CF
        for fam, name, terms_f in ((g.GAUSSIAN, "gaussian", p.terms), (g.LOGISTIC, "logistic", p.terms),
                                   (g.LAPLACE, "laplace", p.terms), (g.CAUCHY, "cauchy", p.terms),
                                   (g.GAUSSIAN, "gaussian, continuous dependency penalty (DEP_CF)", cf_terms)):
            hpf = g.default_hparams(terms=terms_f, family=fam)
            cf = g.Gaus(p, B, hpf)
            sf = cf.new_state(dmu0, dsg0, hpf.lambda0)
            cf.iterate(10, sf)
            sf = cf.new_state(dmu0, dsg0, hpf.lambda0)
            evf = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            n_f = 100
            torch.cuda.synchronize()
            evf[0].record()
            cf.iterate(n_f, sf)
            evf[1].record()
            torch.cuda.synchronize()
            fms = evf[0].elapsed_time(evf[1])
            families.append({"family": name, "iterations": n_f,
                             "restart_iterations_per_s": n_f * B / (fms / 1e3),
                             "ms_per_iteration": fms / n_f,
                             "mean_loss_after": float(sf["loss"].mean().item())})
            cf.close()

    # ---- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        h_mu = torch.from_numpy(mu0.copy()).pin_memory()
        h_sg = torch.from_numpy(sg0.copy()).pin_memory()
        h_mu_out = torch.empty_like(h_mu).pin_memory()
        h_sg_out = torch.empty_like(h_sg).pin_memory()
        h_sched = torch.empty((p.V, B), dtype=torch.int32).pin_memory()
        h_rep = torch.empty(B * 200, dtype=torch.uint8).pin_memory()
        h_loss = torch.empty(B, dtype=torch.float32).pin_memory()
        eev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        torch.cuda.synchronize()
        for k in range(args.steps):
            flush.fill_(k & 255)
            eev[k][0].record()
            init_state(h_mu, h_sg)                   # host -> device copies of the solve's inputs
            solve()
            h_mu_out.copy_(st["mu"], non_blocking=True)
            h_sg_out.copy_(st["sigma"], non_blocking=True)
            h_sched.copy_(sched, non_blocking=True)
            h_rep.copy_(rep, non_blocking=True)
            h_loss.copy_(st["loss"], non_blocking=True)
            eev[k][1].record()
        torch.cuda.synchronize()
        ems = max_over_ranks(sum(a.elapsed_time(b) for a, b in eev), world, dist, "cuda")
        h2d = 2 * p.V * B * 4
        d2h = 2 * p.V * B * 4 + p.V * B * 4 + B * 200 + B * 4
        e2e = {"value": units / (ems / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(p, B, mu0, sg0, hp)

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                "data": "synthetic (seeded logic-network DAG and initial means)",
                "config": dict(describe(p, B, iters, period), l2="flushed between steps (256 MB write)",
                               parallelism=f"restarts sharded, {world} replica(s)"),
                "e2e": e2e, "gpu_launches": args.steps * launches_per_step,
                "clocks": clocks,
                "roofline": {"bound": "alu", "kernel": "k_edges (edge pass)", "achieved": achieved,
                             "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
                             "peak_note": "FP32: 152 SM x 128 lanes x 2 flop x 2070 MHz (max SM clock)",
                             "cost_model": "8 flop per edge-bin (edge pass)",
                             "edge_bins_per_iter": neb_total / iters,
                             "node_pass": {"kernel": "k_nodes", "achieved": nodes_achieved,
                                           "frac": nodes_achieved / peak,
                                           "cost_model": "20 flop per CDF point",
                                           "points_per_iter": npt_total / iters}},
                "iteration_roofline": {
                    "model": "per iteration T* = max(48 V B + (2E + 6V) 4 bytes / HBM, points / SFU exp2, "
                             "(20 points + 8 edge-bins) flop / FP32), summed over the solve's iterations",
                    "t_star_ms_per_step": t_star * 1e3,
                    "t_measured_ms_per_step": ms / args.steps - nchunk * legalize_verify_ms,
                    "frac": t_star * 1e3 / (ms / args.steps - nchunk * legalize_verify_ms),
                    "binding_iterations": t_star_by,
                    "peaks": {"fp32_tflops_measured": fp32_peak / 1e12, "sfu_ex2_per_s_measured": ex2_peak,
                              "hbm_gbs": hbm_peak / 1e9,
                              "fp32_tflops_nominal": peak}},
                "phase_ms_per_iteration": {"k_nodes": ph_ms[0], "k_edges": ph_ms[1],
                                           "reduce_finalize": ph_ms[2], "k_update": ph_ms[3],
                                           "k_edges_first_period": fwd_first, "k_edges_last_period": fwd_last},
                "legalize_verify_ms": legalize_verify_ms,
                "steady_fixed_sigma": steady,
                "solver": solver,
                "formulation_c_sweep": sweep,
                "cdf_families": families,
                "step_ms": step_ms,
                "status_ok": status_ok, "legalized_ok": feasible, "wall_s": wall,
                "cpu_baseline": cpu}
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def phase_probe(args):
    """Iterations 0..N-1 and then iteration N of the benchmark workload, launched
    kernel by kernel (k_nodes, k_edges, k_reduce, k_finalize, k_update each once per
    iteration), so that `ncu -k regex:k_edges -s N -c 1` captures iteration N."""
    import torch

    import paper_2602_20427_gb300 as g
    g.build()
    p, B, mu0, sg0 = workload(0)
    ctx = g.Gaus(p, B, g.default_hparams(terms=p.terms))
    st = ctx.new_state(torch.from_numpy(mu0).cuda(), torch.from_numpy(sg0).cuda())
    if args.phase_probe > 0:
        ctx.profile_iterate(args.phase_probe, st)
    ms = ctx.profile_iterate(1, st)
    torch.cuda.synchronize()
    print(json.dumps({"iteration": args.phase_probe, "phase_ms": {"k_nodes": ms[0], "k_edges": ms[1],
                                                                  "reduce_finalize": ms[2], "k_update": ms[3]}}))
    ctx.close()


def _oracle_iteration(op, ohp, mu, sg, lam, mom, step, lr):
    import oracle
    loss, terms, gm, gs = oracle.loss_grad(op, ohp, mu, sg, lam)
    for th, gg, m1, v1 in ((mu, gm, mom[0], mom[1]), (sg, gs, mom[2], mom[3])):
        flat_t, flat_m, flat_v = th.reshape(-1), m1.reshape(-1), v1.reshape(-1)
        oracle.adam(flat_t, np.ascontiguousarray(gg.reshape(-1)), flat_m, flat_v, step, lr)
    np.maximum(sg, 0.05, out=sg)
    lam[:, 0] += 1e-4 * terms[:, oracle.T_VDEP]
    lam[:, 1] += 1e-4 * terms[:, oracle.T_VRES]


def cpu_baseline(p, B, mu0, sg0, hp, budget_s=12.0, restarts=None):
    """The fp64 oracle, as it stands, on a bounded sample of the same workload."""
    import oracle
    cores = os.cpu_count() or 1
    os.environ.setdefault("OMP_NUM_THREADS", str(cores))
    r = restarts or min(B, cores)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=hp.tau, rho=hp.rho, alpha=hp.alpha, w_res=hp.w_res, w_mem=hp.w_mem, terms=p.terms)
    mu = mu0[:, :r].astype(np.float64).copy()
    sg = sg0[:, :r].astype(np.float64).copy()
    lam = np.full((r, 3), 1e-6)
    mom = [np.zeros_like(mu) for _ in range(4)]
    t0 = time.perf_counter()
    it = 0
    while True:
        it += 1
        _oracle_iteration(op, ohp, mu, sg, lam, mom, it, hp.lr)
        el = time.perf_counter() - t0
        if el >= budget_s or it >= 5:
            break
    return {"value": r * it / el, "unit": UNIT, "cores": int(os.environ.get("OMP_NUM_THREADS", cores)),
            "kind": "oracle", "sample": f"{it} iteration(s) of {r} restarts of {p.name}, fp64, unwindowed, "
                                         f"{el:.1f} s"}


def reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    oracle.build()
    p, B, mu0, sg0 = workload(0)

    class H:  # the same hyperparameters as the GPU arm
        tau, rho, alpha, w_res, w_mem, lr = 1e-2, 1e-4, 1.0, 1.0, 1.0, 1e-2

    cores = os.cpu_count() or 1
    os.environ.setdefault("OMP_NUM_THREADS", str(cores))
    r = min(B, cores)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=H.tau, rho=H.rho, alpha=H.alpha, w_res=H.w_res, w_mem=H.w_mem, terms=p.terms)
    mu = mu0[:, :r].astype(np.float64).copy()
    sg = sg0[:, :r].astype(np.float64).copy()
    lam = np.full((r, 3), 1e-6)
    mom = [np.zeros_like(mu) for _ in range(4)]
    for w in range(args.warmup):
        _oracle_iteration(op, ohp, mu, sg, lam, mom, w + 1, H.lr)
    t0 = time.perf_counter()
    for k in range(args.steps):
        _oracle_iteration(op, ohp, mu, sg, lam, mom, args.warmup + k + 1, H.lr)
    el = time.perf_counter() - t0
    value = args.steps * r / el
    sample = f"1 iteration of {r} of the {B} restarts per step, fp64 oracle, unwindowed"
    print(json.dumps({"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 1,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                      "data": "synthetic (seeded logic-network DAG and initial means)",
                      "config": dict(describe(p, B, args.iters, args.period), sample=sample),
                      "cpu_baseline": {"value": value, "unit": UNIT, "cores": int(os.environ["OMP_NUM_THREADS"]),
                                       "kind": "oracle", "sample": sample},
                      "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


if __name__ == "__main__":
    a = parse()
    if a.phase_probe is not None:
        phase_probe(a)
    elif a.impl == "reference":
        reference_arm(a)
    else:
        gpu_arm(a)
