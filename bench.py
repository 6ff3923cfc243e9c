#!/usr/bin/env python
"""GauS hot-path benchmark: fused loss + gradient + Adam iterations/s x B restarts.

One step = one complete batched solve of Alg. GauS on a workload from its seeded
initial state: the state is initialised (means and deviations copied in, Adam
moments and step zeroed, multipliers set to lambda_0), then the workload's
iterations (gaus_iterate: loss, gradient, Adam, multiplier update; Sec. 3.3) run,
with a round + legalize (App. A) and a verify (Sec. 2.1) of all B restarts every
`--period` iterations.  Every step does the same work, so the number does not
depend on --steps.

`--workload` picks the workload (default: the logic network, V = 10,000, B = 64,
2,000 iterations, the headline); the default run also reports one timed solve of
every other workload under "workloads".  Prints one JSON line.  `--impl reference`
times the fp64 CPU oracle on the same workload and metric (bounded sample per step).
"""
from __future__ import annotations

import argparse
import hashlib
import json
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
SM_MAX_MHZ = 2070.0
PERIOD = 100

# name -> (generator, description); the problem carries its B, iterations, lr and terms
WORKLOADS = {
    "tiny": (lambda: W.tiny_layered(1),
             "tiny layered random DAG: V=64 in 8 layers, 1-3 predecessors, 2 classes (limits 2, 3), "
             "latencies 1..3, D=1.5 critical path, B=1, 200 iterations at lr 0.05"),
    "random": (lambda: W.random_layered(1),
               "random layered DAG: V=1,000, depth ~40, Poisson fan-in 2, 4 classes (limits 8/6/4/2), "
               "latencies 1..4, D=1.5 critical path, B=64, 1,000 iterations"),
    "logic": (lambda: W.logic_network(1),
              "AND/INV logic network: V=10,000, depth 120, Zipf fan-out capped at 64, 2 classes "
              "(AND limit 64, INV unlimited), unit latency, D=1.3 depth, B=64, 2,000 iterations"),
    "modulo_mii": (lambda: W.modulo_loop(1, ii_factor=1.0),
                   "loop body (Formulation C): V=5,000, ~8,000 edges + 200 back edges (distance 1..3), "
                   "6 classes (limits 2-16), latencies 1..6, II=MII, D=3 II, B=32, 2,000 iterations"),
    "modulo_1.25mii": (lambda: W.modulo_loop(1, ii_factor=1.25),
                       "loop body (Formulation C) at II=1.25 MII, D=3 II, B=32, 2,000 iterations"),
    "modulo_1.5mii": (lambda: W.modulo_loop(1, ii_factor=1.5),
                      "loop body (Formulation C) at II=1.5 MII, D=3 II, B=32, 2,000 iterations"),
    "wide": (lambda: W.wide_layered(1),
             "wide streaming-processor DAG: V=50,000 (width 1,000, depth 50), 2-4 predecessors from the "
             "previous 1-3 layers, 8 classes (limit 128), latencies 1..8, register-lifetime term, "
             "D=1.4 critical path, B=16, 2,000 iterations"),
}
HEADLINE = "logic"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default=HEADLINE, choices=sorted(WORKLOADS))
    ap.add_argument("--iters", type=int, default=None, help="iterations per solve (default: the workload's)")
    ap.add_argument("--period", type=int, default=PERIOD, help="iterations between legalize + verify")
    ap.add_argument("--impl", default="gaus", choices=["gaus", "reference"])
    ap.add_argument("--phase-probe", type=int, default=None, metavar="N",
                    help="run N iterations kernel by kernel, then one more, print the phase times and exit "
                         "(a fixed launch sequence for ncu captures at iteration N)")
    ap.add_argument("--fused-probe", type=int, default=None, metavar="N",
                    help="run N fused iterations, then one gaus_iterate call of --period iterations between "
                         "cudaProfilerStart/Stop, and exit (for ncu captures of one k_fused launch)")
    ap.add_argument("--cpu-sample", default=None, metavar="WORKLOAD",
                    help="internal: time the oracle on a bounded sample of WORKLOAD and print one JSON line")
    ap.add_argument("--threads", type=int, default=None, help="with --cpu-sample: oracle threads")
    ap.add_argument("--budget", type=float, default=12.0, help="with --cpu-sample: seconds of oracle work")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-solver", action="store_true", help="skip the complete-solver runs (gaus_solve)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-families", action="store_true", help="skip the CDF-family timings")
    ap.add_argument("--no-workloads", action="store_true", help="skip the other workloads' timed solves")
    ap.add_argument("--path", default="auto", choices=["auto", "fused", "multi"],
                    help="gaus_iterate's path: chosen per call (default), or forced")
    ap.add_argument("--restarts", type=int, default=None,
                    help="restarts per rank (default: the workload's B; others for scaling studies)")
    ap.add_argument("--profile-range", action="store_true",
                    help="bracket the timed steps with cudaProfilerStart/Stop (for ncu --profile-from-start off)")
    return ap.parse_args()


def make_workload(name):
    p = WORKLOADS[name][0]()
    return p


def workload(rank=0, B=None, name=HEADLINE):
    """The benchmark workload of one rank: the same DAG on every rank, and B
    restarts of its own (initial state seeded by the rank), so the ranks' restarts
    are independent and need no data-path collective (weak scaling)."""
    p = make_workload(name)
    B = p.B if B is None else B
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


def describe(name, p, B, iters, period=None):
    d = {"workload": f"{p.name}: {WORKLOADS[name][1]}", "B": B, "V": p.V, "E": p.E, "D": p.D,
         "iterations_per_step": iters, "legalize_verify_every": period,
         "init": "mu = earliest start + N(0, 2), sigma = 1.5 (seeded)", "lr": p.lr, "window_k": 6.0,
         "terms": p.terms}
    if p.II:
        d.update(II=p.II, back_edges=p.NB)
    return d


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
def algorithmic_work(torch, mu, sg, src, dst, k, D, storage=False):
    """The design-independent work of one iteration, from the +-k sigma windows:
    window points (one CDF evaluation, one exp each), edge-bins (dependency edge:
    producer bins; communication: producer + consumer bins) and, with the storage
    term, storage point-edges (every point of a consumer's window paired with each
    of its producers: one factor of the product 1 - M).  A window of n points covers
    n + 1 bins.  Returns (fp32 flop, points, edge-bins, storage point-edges) under the
    cost model of 20 flop per point and 8 per edge-bin or storage point-edge."""
    a = torch.clamp(torch.ceil(mu - k * sg - 0.5), 0, D - 1)
    b = torch.clamp(torch.floor(mu + k * sg - 0.5), -1, D - 2)
    bins = (b - a + 2).to(torch.float64)                  # (V, B)
    n_pt = float(bins.sum())
    n_eb = float((2.0 * bins[src] + bins[dst]).sum())
    n_st = float((bins[dst] - 1.0).sum()) if storage else 0.0
    return 20.0 * n_pt + 8.0 * (n_eb + n_st), n_pt, n_eb, n_st


def algorithmic_flops(torch, mu, sg, src, dst, k, D):
    """(fp32 flop, points, edge-bins) of one iteration without the storage term."""
    f, n_pt, n_eb, _ = algorithmic_work(torch, mu, sg, src, dst, k, D)
    return f, n_pt, n_eb


def state_bytes(p, B):
    """HBM bytes one iteration must move whatever the design: the state read and
    written (mu, sigma, four Adam moments: 48 V B) and the graph read once
    ((2E + 6V) 4)."""
    return 48.0 * p.V * B + (2.0 * p.E + 6.0 * p.V) * 4.0


def measured_peaks():
    """MEASURED_PEAKS.json (HBM copy GB/s), else the fallback of an earlier GB300 measurement."""
    try:
        d = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
        return {"hbm_gbs": float(d["hbm_gbs"]), "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "source": "fallback"}


def measured_hbm_gbs():
    return measured_peaks()["hbm_gbs"]


FUSED_PROFILE = os.path.join("profiles", "k_fused_logic_network_v10000_b64.md")
FUSED_SOURCES = ("gaus_fused.cuh", "gaus_device.cuh", "gaus_api.cu", "gaus_plan.cpp")


def source_hash(files=FUSED_SOURCES):
    """sha256 over the sha256sum lines of the kernel's sources (as `sha256sum | sha256sum`)."""
    lines = []
    for f in files:
        path = os.path.join(ROOT, "paper_2602_20427_gb300", "csrc", f)
        h = hashlib.sha256(open(path, "rb").read()).hexdigest()
        lines.append(f"{h}  paper_2602_20427_gb300/csrc/{f}\n")
    return hashlib.sha256("".join(lines).encode()).hexdigest()


def profiled_traffic():
    """DRAM bytes per k_fused launch of the headline workload from the committed ncu
    summary, or None when the kernel's sources changed since that capture."""
    prof = os.path.join(ROOT, FUSED_PROFILE)
    if not os.path.exists(prof):
        return None
    want = {}
    for line in open(prof).read().splitlines():
        if ":" in line and line.split(":")[0] in ("dram-bytes-per-launch", "source-sha256"):
            want[line.split(":")[0]] = line.split(":", 1)[1].strip()
    if want.get("source-sha256") != source_hash() or "dram-bytes-per-launch" not in want:
        return None
    return float(want["dram-bytes-per-launch"])


# ----------------------------------------------------------------- one solve = one step
class Solve:
    """One step of a workload: the state initialised from (mu, sigma), then `iters`
    fused iterations with a legalize + verify of all restarts every `period`."""

    def __init__(self, torch, ctx, p, B, hp, iters, period):
        self.ctx, self.hp, self.iters, self.period = ctx, hp, iters, period
        dev = "cuda"
        self.st = ctx.new_state(torch.zeros((p.V, B), device=dev), torch.ones((p.V, B), device=dev), hp.lambda0)
        self.sched = torch.empty((p.V, B), dtype=torch.int32, device=dev)
        self.lstat = torch.empty(B, dtype=torch.int32, device=dev)
        self.rep = torch.empty(B * 200, dtype=torch.uint8, device=dev)

    def init(self, mu_src, sg_src):
        st = self.st
        st["mu"].copy_(mu_src, non_blocking=True)
        st["sigma"].copy_(sg_src, non_blocking=True)
        for kk in ("m_mu", "v_mu", "m_sigma", "v_sigma", "loss", "terms"):
            st[kk].zero_()
        st["step"].zero_()
        st["status"].zero_()
        st["lambda_"].fill_(self.hp.lambda0)

    def solve(self):
        for _ in range(self.iters // self.period):
            self.ctx.iterate(self.period, self.st)
            self.ctx.legalize(self.st["mu"], self.sched, self.lstat)
            self.ctx.verify_raw(self.sched, self.rep)

    def step(self, mu_src, sg_src):
        self.init(mu_src, sg_src)
        self.solve()


def launches_per_step(plan, iters, period, fused_calls=None, multi_iters=None, choices=0):
    """Kernel launches of one step: per gaus_iterate call the cooperative k_fused
    launches (fused path) or the per-iteration kernels (multi-kernel path) and, when
    the path is chosen per call, the window reduction of the choice; per period the
    legalization kernel and the verifier's two passes.  Without the counts of a
    measured step, every call is taken to run the plan's preferred path."""
    calls = iters // period
    if fused_calls is None:
        fused_calls = calls if plan["fused"] else 0
        multi_iters = 0 if plan["fused"] else iters
    return (fused_calls * plan["fused_launches_per_call"] + multi_iters * plan["launches_per_iteration"]
            + choices + calls * 3)


def path_counts(ctx):
    i = ctx.plan_info()
    return i["fused_calls"], i["multi_iterations"], i["path_choices"]


def device_peaks(g, torch):
    """This device's FP32 FMA and SFU exp2 throughput (the library's microbenchmark),
    the HBM copy bandwidth of MEASURED_PEAKS.json and the device's SM count."""
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    hb = measured_peaks()
    return {"fp32": g.measure_peak(g.PEAK_FP32), "ex2": g.measure_peak(g.PEAK_EX2),
            "hbm": hb["hbm_gbs"] * 1e9, "hbm_source": hb["source"], "sms": int(props.multi_processor_count)}


def iteration_roofline(torch, ctx, solve, p, B, hp, mu0, sg0, peaks, plan):
    """Run one solve's iterations (no legalize) call by call from the initial state,
    timing each gaus_iterate call of `period` iterations with CUDA events, and the
    design-independent work at the start and end of each call.  Per iteration
    T* = max(state bytes / HBM, points / SFU exp2, flop / FP32); the roofline of the
    dominant kernel (k_fused, one launch per call, on the fused path; the iteration's
    kernel sequence otherwise) takes the resource with the largest share of T*."""
    solve.init(mu0, sg0)
    st = solve.st
    src = torch.from_numpy(np.asarray(p.src, np.int64)).cuda()
    dst = torch.from_numpy(np.asarray(p.dst, np.int64)).cuda()
    storage = bool(p.terms & W.REG_OBJ)
    period, nchunk = solve.period, solve.iters // solve.period
    sb = state_bytes(p, B)
    tot = {"flop": 0.0, "points": 0.0, "edge_bins": 0.0, "storage_pe": 0.0, "bytes": 0.0, "t": 0.0,
           "t_star": 0.0, "alg_t": {"hbm": 0.0, "sfu": 0.0, "fp32": 0.0}}
    binding = {"hbm": 0, "sfu": 0, "fp32": 0}
    ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    calls_ms = []
    w0 = algorithmic_work(torch, st["mu"], st["sigma"], src, dst, hp.window_k, p.D, storage)
    fused_t, fused_bytes, fused_flop, fused_pts, fused_calls = 0.0, 0.0, 0.0, 0.0, 0
    for _ in range(nchunk):
        f0 = path_counts(ctx)[0]
        torch.cuda.synchronize()
        ev[0].record()
        ctx.iterate(period, st)
        ev[1].record()
        torch.cuda.synchronize()
        ms = ev[0].elapsed_time(ev[1])
        calls_ms.append(ms)
        was_fused = path_counts(ctx)[0] > f0
        w1 = algorithmic_work(torch, st["mu"], st["sigma"], src, dst, hp.window_k, p.D, storage)
        fl, pt, eb, sp = (0.5 * (x + y) for x, y in zip(w0, w1))
        w0 = w1
        alg = {"hbm": sb / peaks["hbm"], "sfu": pt / peaks["ex2"], "fp32": fl / peaks["fp32"]}
        for k in alg:
            tot["alg_t"][k] += period * alg[k]
        tot["t_star"] += period * max(alg.values())
        binding[max(alg, key=alg.get)] += period
        tot["flop"] += period * fl
        tot["points"] += period * pt
        tot["edge_bins"] += period * eb
        tot["storage_pe"] += period * sp
        tot["bytes"] += period * sb
        tot["t"] += ms * 1e-3
        if was_fused:
            fused_calls += 1
            fused_t += ms * 1e-3
            fused_bytes += period * sb
            fused_flop += period * fl
            fused_pts += period * pt
    res = max(tot["alg_t"], key=tot["alg_t"].get)
    # the dominant kernel: k_fused over the calls it ran, when it ran any
    kt, kb, kf, kp = (fused_t, fused_bytes, fused_flop, fused_pts) if fused_calls else \
        (tot["t"], tot["bytes"], tot["flop"], tot["points"])
    if res == "hbm":
        achieved, peak, unit, bound = kb / kt / 1e9, peaks["hbm"] / 1e9, "GB/s", "hbm"
        pk_note = f"HBM copy bandwidth ({peaks['hbm_source']}, MEASURED_PEAKS.json)"
    elif res == "sfu":
        achieved, peak, unit, bound = kp / kt / 1e9, peaks["ex2"] / 1e9, "Gexp2/s", "alu"
        pk_note = "SFU exp2 results/s, measured on this device (gaus_measure_peak)"
    else:
        achieved, peak, unit, bound = kf / kt / 1e12, peaks["fp32"] / 1e12, "TFLOP/s", "alu"
        pk_note = "FP32 FMA throughput, measured on this device (gaus_measure_peak)"
    iters = nchunk * period
    kernel = "k_fused" if fused_calls else "iteration kernel sequence (k_nodes .. k_update" + \
        (", k_reg_fwd, k_reg_bwd)" if storage else ")")
    roof = {"bound": bound, "kernel": kernel, "achieved": achieved, "peak": peak, "unit": unit,
            "frac": achieved / peak, "peak_note": pk_note + " (of measured)",
            "calls": {"fused": fused_calls, "multi_kernel": nchunk - fused_calls},
            "launches": fused_calls * plan["fused_launches_per_call"] if fused_calls else
            nchunk * period * plan["launches_per_iteration"],
            "mean_launch_ms": fused_t * 1e3 / fused_calls if fused_calls else None,
            "cost_model": "20 flop and 1 exp2 per window point, 8 flop per edge-bin and per storage "
                          "point-edge; 48 V B + (2E + 6V) 4 state bytes per iteration",
            "per_iteration": {"points": tot["points"] / iters, "edge_bins": tot["edge_bins"] / iters,
                              "storage_point_edges": tot["storage_pe"] / iters, "state_bytes": sb}}
    it_roof = {"model": "per iteration T* = max(state bytes / HBM, points / SFU exp2, flop / FP32), "
                        "summed over the solve's iterations; T = CUDA-event time of the gaus_iterate calls",
               "t_star_ms": tot["t_star"] * 1e3, "t_ms": tot["t"] * 1e3, "frac": tot["t_star"] / tot["t"],
               "binding_iterations": binding, "us_per_iteration": tot["t"] * 1e6 / iters,
               "us_per_iteration_first_call": calls_ms[0] * 1e3 / period,
               "us_per_iteration_last_call": calls_ms[-1] * 1e3 / period,
               "peaks": {"fp32_tflops": peaks["fp32"] / 1e12, "sfu_gexp2_per_s": peaks["ex2"] / 1e9,
                         "hbm_gbs": peaks["hbm"] / 1e9, "sms": peaks["sms"],
                         "fp32_tflops_nominal": peaks["sms"] * FP32_LANES_PER_SM * 2 * SM_MAX_MHZ * 1e6 / 1e12}}
    return roof, it_roof


def fused_phases(torch, g, p, B, hp, mu0, sg0, marks=(0, 100, 1500)):
    """Phase profile of the persistent kernel at a few iterations of the solve (us):
    the slowest block's (critical) and the mean block's time in each phase, the two
    group-barrier latencies and the iteration (gaus_profile_phases, 10 iterations)."""
    ctx = g.Gaus(p, B, hp)
    st = ctx.new_state(mu0, sg0, hp.lambda0)
    out, done = {}, 0
    for mk in marks:
        if mk >= p.iters:
            break
        if mk > done:
            ctx.iterate(mk - done, st)
        ph = ctx.profile_phases(10, st)
        done = mk + 10
        out[f"iteration_{mk}"] = {k: round(v * 1e3, 2) for k, v in ph.items()}
    ctx.close()
    return out


# ----------------------------------------------------------------- Formulation C feasibility witness
def modulo_list_schedule(p, max_rounds=30):
    """A feasibility witness for a loop body at its II (not part of GauS): greedy
    modulo list scheduling in topological order -- each node at the earliest step
    that meets its forward edges and its lower bound, has a free slot of its class
    in the modulo reservation table (demand counted at the start step, folded mod
    II) and ends by D -- repeated with the lower bound of a back edge's head raised
    while that back edge (s_i + dist II >= s_j + Lat_j) is violated.  Returns the
    schedule (int32, V) or None when no round meets every constraint; a schedule is
    a witness only once gaus_verify accepts it, and None proves nothing."""
    V, II, D = p.V, int(p.II), int(p.D)
    src, dst = np.asarray(p.src, np.int64), np.asarray(p.dst, np.int64)
    if II <= 0 or np.any(src >= dst):
        return None
    lat, cls = np.asarray(p.lat, np.int64), np.asarray(p.cls, np.int64)
    dem = np.asarray(p.demand, np.int64)
    lim = [np.inf if not np.isfinite(x) else int(x) for x in np.asarray(p.limit, np.float64)]
    preds = [[] for _ in range(V)]
    for u, v in zip(src.tolist(), dst.tolist()):
        preds[v].append(u)
    lb = np.zeros(V, np.int64)
    for _ in range(max_rounds):
        mrt = np.zeros((p.C, II), np.int64)
        s = np.zeros(V, np.int64)
        placed = True
        for v in range(V):
            t0 = int(lb[v])
            for u in preds[v]:
                t0 = max(t0, int(s[u] + lat[u]))
            c, last = int(cls[v]), D - int(lat[v])
            t = t0
            while t <= min(t0 + II - 1, last) and mrt[c, t % II] + dem[v] > lim[c]:
                t += 1
            if t > min(t0 + II - 1, last):
                placed = False
                break
            s[v] = t
            mrt[c, t % II] += dem[v]
        if not placed:
            return None
        raised = False
        for j, i, dist in zip(np.asarray(p.bsrc).tolist(), np.asarray(p.bdst).tolist(),
                              np.asarray(p.bdist).tolist()):
            need = int(s[j] + lat[j] - dist * II)
            if s[i] < need:
                lb[i] = max(lb[i], need)
                raised = True
        if not raised:
            return s.astype(np.int32)
    return None


# ----------------------------------------------------------------- GPU arm
def timed_steps(torch, solve, mu_src, sg_src, steps, flush, profile_range=False):
    """`steps` steps bracketed by CUDA events, the L2 flushed (256 MB write) before each."""
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    if profile_range:
        torch.cuda.profiler.start()              # ncu --profile-from-start off: the timed steps only
    for k in range(steps):
        flush.fill_(k & 255)
        evs[k][0].record()
        solve.step(mu_src, sg_src)
        evs[k][1].record()
    torch.cuda.synchronize()
    if profile_range:
        torch.cuda.profiler.stop()
    return [a.elapsed_time(b) for a, b in evs]


def other_workload(torch, g, name, peaks, flush):
    """One timed solve (after one untimed) of another workload, its iteration roofline
    and how many restarts end legal without resource overflow."""
    p, B, mu0, sg0 = workload(0, None, name)
    hp = g.default_hparams(terms=p.terms, lr=p.lr)
    ctx = g.Gaus(p, B, hp)
    plan = ctx.plan_info()
    period = min(PERIOD, p.iters)
    S = Solve(torch, ctx, p, B, hp, p.iters, period)
    dmu0, dsg0 = torch.from_numpy(mu0).cuda(), torch.from_numpy(sg0).cuda()
    S.step(dmu0, dsg0)
    torch.cuda.synchronize()
    c0 = path_counts(ctx)
    ms = timed_steps(torch, S, dmu0, dsg0, 1, flush)[0]
    c1 = path_counts(ctx)
    rep = ctx.verify(S.sched)
    ok = int(sum(1 for r in rep if r["feasible"] and r["res_ok"]))
    roof, it_roof = iteration_roofline(torch, ctx, S, p, B, hp, dmu0, dsg0, peaks, plan)
    ctx.close()
    return {"config": describe(name, p, B, p.iters, period), "value": p.iters * B / (ms / 1e3), "unit": UNIT,
            "ms_per_step": ms,
            "calls": {"fused": c1[0] - c0[0], "multi_kernel": p.iters // period - (c1[0] - c0[0])},
            "gpu_launches_per_step": launches_per_step(plan, p.iters, period, c1[0] - c0[0], c1[1] - c0[1],
                                                       c1[2] - c0[2]),
            "roofline": {k: roof[k] for k in ("bound", "kernel", "achieved", "peak", "unit", "frac")},
            "iteration_roofline": {k: it_roof[k] for k in ("t_star_ms", "t_ms", "frac", "us_per_iteration",
                                                           "us_per_iteration_last_call", "binding_iterations")},
            "restarts_legal_without_overflow_at_end": ok}


def formulation_c_sweep(torch, g, n_periods=40, period=PERIOD):
    """Formulation C at II in {MII, 1.25 MII, 1.5 MII} on the loop body: a feasibility
    witness from modulo list scheduling checked by gaus_verify, and the complete
    solver (gaus_solve) from the workload's initialization for n_periods x period
    iterations: how many restarts reach a legal best without resource overflow, and
    the iteration of the first."""
    out = []
    for factor in (1.0, 1.25, 1.5):
        pm = W.modulo_loop(1, ii_factor=factor)
        Bm = pm.B
        mu_m, sg_m = W.init_state(pm, Bm, seed=1)
        hpm = g.default_hparams(terms=pm.terms)
        cm = g.Gaus(pm, Bm, hpm)
        wit = modulo_list_schedule(pm)
        witness = None
        if wit is not None:
            rep = cm.verify(torch.from_numpy(np.repeat(wit[:, None], Bm, axis=1)).cuda())[0]
            witness = {"found": bool(rep["feasible"] and rep["res_ok"]), "L_mmem": rep["L_mmem"],
                       "score": hpm.w_mem * rep["L_mmem"], "peak_usage": rep["peak"]}
        mu_d = torch.from_numpy(mu_m).cuda()

        def init_m(out=None):
            b = cm.init_state(kappa=1.0 / 6.0, mu0=mu_d, out=out)
            b[0]["sigma"].fill_(float(sg_m[0, 0]))
            b[1].fill_(float(sg_m[0, 0]))
            return b

        bm = init_m()
        wm = cm.solve(1, period, *bm)                 # captures the graphs
        init_m(out=bm)
        ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        torch.cuda.synchronize()
        ev[0].record()
        cm.solve(n_periods, period, *bm, work=wm)
        ev[1].record()
        torch.cuda.synchronize()
        ms = ev[0].elapsed_time(ev[1])
        sc = bm[2]["score"].cpu().numpy()
        it = bm[2]["iter"].cpu().numpy()
        fnd = np.isfinite(sc)
        ls = wm["leg_status"].cpu().numpy()
        out.append({"ii_factor": factor, "II": pm.II, "MII": int(pm.mii), "D": pm.D, "V": pm.V, "E": pm.E,
                    "back_edges": pm.NB, "B": Bm, "iterations": n_periods * period,
                    "restart_iterations_per_s": n_periods * period * Bm / (ms / 1e3),
                    "list_schedule_witness": witness,
                    "restarts_with_feasible_best": int(fnd.sum()),
                    "first_feasible_best_at_iteration": int(it[fnd].min()) if fnd.any() else None,
                    "best_score_min": float(sc[fnd].min()) if fnd.any() else None,
                    "best_score_mean": float(sc[fnd].mean()) if fnd.any() else None,
                    "last_legalize_not_converged": int((ls == 7).sum()),
                    "init": "mu = earliest start + N(0, 2), sigma = 1.5 (seeded)",
                    "score": "w_mem L_mmem of the best legal schedule (no resource overflow)"})
        cm.close()
    return out


def complete_solver(torch, g, p, B, hp, dmu0, dsg0, iters, period):
    """The outer loop of Alg. GauS on the device (gaus_solve): one solve of the
    step's length from the kappa initialization, and one twice as long from the
    timed workload's initialization (anytime quality)."""
    ctxS = g.Gaus(p, B, hp)
    bufs = ctxS.init_state(kappa=1.0 / 6.0)
    work = ctxS.solve(1, period, *bufs)                    # captures the graphs
    ctxS.init_state(kappa=1.0 / 6.0, out=bufs)
    ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    torch.cuda.synchronize()
    ev[0].record()
    ctxS.solve(iters // period, period, *bufs, work=work)
    ev[1].record()
    torch.cuda.synchronize()
    sms = ev[0].elapsed_time(ev[1])
    bsc = bufs[2]["score"].cpu().numpy()
    found = np.isfinite(bsc)
    solver = {"value": iters * B / (sms / 1e3), "unit": UNIT, "ms": sms,
              "init": "kappa = 1/6: sigma = max(kappa (ALAP - ASAP), sigma_min), mu = (ASAP + ALAP) / 2",
              "periods": iters // period, "period": period,
              "restarts_with_feasible_best": int(found.sum()),
              "best_score_min": float(bsc[found].min()) if found.any() else None,
              "best_score_mean": float(bsc[found].mean()) if found.any() else None,
              "score": "L_res + alpha L_com of the best legal schedule (no resource overflow)"}
    bufs = ctxS.init_state(kappa=1.0 / 6.0, mu0=dmu0, out=bufs)
    bufs[0]["sigma"].copy_(dsg0)
    bufs[1].copy_(dsg0)
    n_long = 2 * iters // period
    torch.cuda.synchronize()
    ev[0].record()
    ctxS.solve(n_long, period, *bufs, work=work)
    ev[1].record()
    torch.cuda.synchronize()
    lms = ev[0].elapsed_time(ev[1])
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
    return solver


def cdf_families(torch, g, p, B, dmu0, dsg0, n_f=100):
    """App. D: the first n_f fused iterations of the workload from the same
    initialization with the normal, logistic, Laplace and Cauchy relaxations (heavier
    tails: wider windows), and the normal with the continuous dependency penalty in
    place of the binned Eq. dep."""
    families = []
    cf_terms = (p.terms & ~g.DEP) | g.DEP_CF
    for fam, name, terms_f in ((g.GAUSSIAN, "gaussian", p.terms), (g.LOGISTIC, "logistic", p.terms),
                               (g.LAPLACE, "laplace", p.terms), (g.CAUCHY, "cauchy", p.terms),
                               (g.GAUSSIAN, "gaussian, continuous dependency penalty (DEP_CF)", cf_terms)):
        hpf = g.default_hparams(terms=terms_f, family=fam, lr=p.lr)
        cf = g.Gaus(p, B, hpf)
        sf = cf.new_state(dmu0, dsg0, hpf.lambda0)
        cf.iterate(10, sf)
        sf = cf.new_state(dmu0, dsg0, hpf.lambda0)
        f0 = path_counts(cf)[0]
        ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        torch.cuda.synchronize()
        ev[0].record()
        cf.iterate(n_f, sf)
        ev[1].record()
        torch.cuda.synchronize()
        fms = ev[0].elapsed_time(ev[1])
        families.append({"family": name, "iterations": n_f,
                         "path": "fused" if path_counts(cf)[0] > f0 else "multi-kernel",
                         "restart_iterations_per_s": n_f * B / (fms / 1e3),
                         "ms_per_iteration": fms / n_f, "mean_loss_after": float(sf["loss"].mean().item())})
        cf.close()
    return families


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
    name = args.workload
    headline = name == HEADLINE
    p, B, mu0, sg0 = workload(rank, args.restarts, name)
    iters = args.iters or p.iters
    period = min(args.period, iters)
    assert iters % period == 0, "--iters must be a multiple of --period"
    hp = g.default_hparams(terms=p.terms, lr=p.lr)
    ctx = g.Gaus(p, B, hp)
    ctx.set_path({"auto": g.PATH_AUTO, "fused": g.PATH_FUSED, "multi": g.PATH_MULTI}[args.path])
    plan = ctx.plan_info()
    dmu0, dsg0 = torch.from_numpy(mu0).cuda(), torch.from_numpy(sg0).cuda()
    S = Solve(torch, ctx, p, B, hp, iters, period)
    for _ in range(args.warmup):
        S.step(dmu0, dsg0)
    torch.cuda.synchronize()
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device="cuda")
    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(local).uuid)
    except Exception:
        gpu_id = None
    peaks = device_peaks(g, torch)
    sampler = ClockSampler(gpu_id) if rank == 0 else None
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
        time.sleep(0.5)
    wall0 = time.perf_counter()
    c0 = path_counts(ctx)
    step_ms = timed_steps(torch, S, dmu0, dsg0, args.steps, flush, args.profile_range)
    c1 = path_counts(ctx)
    wall = time.perf_counter() - wall0
    # our kernels in the timed region: each call's path as the library counted it
    df, dm, dc = (b - a for a, b in zip(c0, c1))
    launches = (df * plan["fused_launches_per_call"] + dm * plan["launches_per_iteration"] + dc
                + args.steps * (iters // period) * 3)
    clocks = sampler.stop() if sampler else None
    ms = sum(step_ms)
    if world > 1:
        dist.barrier()
    ms = max_over_ranks(ms, world, dist, "cuda")
    status_ok = bool(int(S.st["status"].abs().sum()) == 0)
    legal = int((S.lstat == 0).sum())
    value = job_throughput(args.steps, iters, B, world, ms)

    # ---- legalize + verify alone (part of every step above; reported separately)
    lv = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    lv[0].record()
    for _ in range(10):
        ctx.legalize(S.st["mu"], S.sched, S.lstat)
        ctx.verify_raw(S.sched, S.rep)
    lv[1].record()
    torch.cuda.synchronize()
    legalize_verify_ms = lv[0].elapsed_time(lv[1]) / 10

    # ---- roofline: the solve's iterations call by call, with the algorithmic work
    roof, it_roof = iteration_roofline(torch, ctx, S, p, B, hp, dmu0, dsg0, peaks, plan)
    roof["traffic"] = profiled_traffic() if headline and plan["fused"] else None
    phases = fused_phases(torch, g, p, B, hp, dmu0, dsg0) if plan["fused"] and rank == 0 else None

    extra = {}
    if headline and rank == 0:
        # steady state at fixed sigma: the initial state with lr = 1e-20 (an Adam step
        # is at most ~lr, far below one ulp of mu or sigma, so the windows never shrink)
        hp0 = g.default_hparams(terms=p.terms, lr=1e-20)
        ctx0 = g.Gaus(p, B, hp0)
        st0 = ctx0.new_state(dmu0, dsg0, hp0.lambda0)
        ctx0.iterate(20, st0)
        ev0 = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        torch.cuda.synchronize()
        ev0[0].record()
        ctx0.iterate(200, st0)
        ev0[1].record()
        torch.cuda.synchronize()
        fixed_ms = ev0[0].elapsed_time(ev0[1]) / 200
        ctx0.close()
        extra["steady_fixed_sigma"] = {
            "value": B / (fixed_ms / 1e3), "unit": UNIT, "sigma": 1.5, "us_per_iteration": fixed_ms * 1e3,
            "note": "initial state of the same workload with lr = 1e-20, so every iteration has the "
                    "initial +-6 sigma windows (the most expensive point of the run)"}
        if not args.no_solver:
            extra["solver"] = complete_solver(torch, g, p, B, hp, dmu0, dsg0, iters, period)
            extra["formulation_c_sweep"] = formulation_c_sweep(torch, g)
        if not args.no_families:
            extra["cdf_families"] = cdf_families(torch, g, p, B, dmu0, dsg0)
        if not args.no_workloads:
            extra["workloads"] = {n: other_workload(torch, g, n, peaks, flush) for n in WORKLOADS if n != name}

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
            S.step(h_mu, h_sg)                       # host -> device copies of the solve's inputs
            h_mu_out.copy_(S.st["mu"], non_blocking=True)
            h_sg_out.copy_(S.st["sigma"], non_blocking=True)
            h_sched.copy_(S.sched, non_blocking=True)
            h_rep.copy_(S.rep, non_blocking=True)
            h_loss.copy_(S.st["loss"], non_blocking=True)
            eev[k][1].record()
        torch.cuda.synchronize()
        ems = max_over_ranks(sum(a.elapsed_time(b) for a, b in eev), world, dist, "cuda")
        h2d = 2 * p.V * B * 4
        d2h = 2 * p.V * B * 4 + p.V * B * 4 + B * 200 + B * 4
        e2e = {"value": job_throughput(args.steps, iters, B, world, ems), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_sample_subprocess(name, os.cpu_count() or 1, 12.0)
        if cpu is not None:
            cpu["single_thread"] = cpu_sample_subprocess(name, 1, 12.0)

    if rank == 0:
        line = {"metric": METRIC if headline else METRIC.replace("logic-network DAG, |V|=10k", p.name),
                "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                "data": f"synthetic (seeded {p.name} DAG and initial means)",
                "config": dict(describe(name, p, B, iters, period), l2="flushed between steps (256 MB write)",
                               path=args.path,
                               parallelism=f"restarts sharded, {world} replica(s)"),
                "e2e": e2e, "gpu_launches": launches,
                "calls": {"fused": df, "multi_kernel": args.steps * (iters // period) - df},
                "clocks": clocks, "roofline": roof, "iteration_roofline": it_roof,
                "plan": plan, "fused_phases_us": phases,
                "legalize_verify_ms": legalize_verify_ms, "step_ms": step_ms,
                "status_ok": status_ok, "legalized_ok": legal, "wall_s": wall, "cpu_baseline": cpu}
        line.update(extra)
        print(json.dumps(line))
    ctx.close()
    if world > 1:
        dist.destroy_process_group()


def phase_probe(args):
    """Iterations 0..N-1 and then iteration N of the workload, launched kernel by
    kernel, so that `ncu -k regex:<kernel> -s N -c 1` captures iteration N."""
    import torch

    import paper_2602_20427_gb300 as g
    g.build()
    p, B, mu0, sg0 = workload(0, None, args.workload)
    ctx = g.Gaus(p, B, g.default_hparams(terms=p.terms, lr=p.lr))
    st = ctx.new_state(torch.from_numpy(mu0).cuda(), torch.from_numpy(sg0).cuda())
    if args.phase_probe > 0:
        ctx.profile_iterate(args.phase_probe, st)
    ms = ctx.profile_iterate(1, st)
    torch.cuda.synchronize()
    print(json.dumps({"iteration": args.phase_probe, "phase_ms": ms}))
    ctx.close()


def fused_probe(args):
    """N fused iterations of the workload, then one gaus_iterate call of --period
    iterations (one k_fused launch) between cudaProfilerStart/Stop."""
    import torch

    import paper_2602_20427_gb300 as g
    g.build()
    p, B, mu0, sg0 = workload(0, None, args.workload)
    ctx = g.Gaus(p, B, g.default_hparams(terms=p.terms, lr=p.lr))
    ctx.set_path(g.PATH_FUSED)   # the probe is of the fused kernel, whatever the windows
    st = ctx.new_state(torch.from_numpy(mu0).cuda(), torch.from_numpy(sg0).cuda())
    if args.fused_probe > 0:
        ctx.iterate(args.fused_probe, st)
    torch.cuda.synchronize()
    ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    torch.cuda.profiler.start()
    ev[0].record()
    ctx.iterate(args.period, st)
    ev[1].record()
    torch.cuda.synchronize()
    torch.cuda.profiler.stop()
    print(json.dumps({"iteration": args.fused_probe, "iterations": args.period, "plan": ctx.plan_info(),
                      "ms": ev[0].elapsed_time(ev[1]), "status": int(st["status"].abs().sum())}))
    ctx.close()


# ----------------------------------------------------------------- the fp64 oracle on the host cores
# the library's default hyperparameters (gaus_default_hparams), restated so that the
# oracle's side never loads the CUDA library
TAU, RHO, LAMBDA0, ALPHA, W_RES, W_MEM, SIGMA_MIN = 1e-2, 1e-4, 1e-6, 1.0, 1.0, 1.0, 0.05


def _oracle_iteration(op, ohp, mu, sg, lam, mom, step, lr):
    import oracle
    loss, terms, gm, gs = oracle.loss_grad(op, ohp, mu, sg, lam)
    for th, gg, m1, v1 in ((mu, gm, mom[0], mom[1]), (sg, gs, mom[2], mom[3])):
        flat_t, flat_m, flat_v = th.reshape(-1), m1.reshape(-1), v1.reshape(-1)
        oracle.adam(flat_t, np.ascontiguousarray(gg.reshape(-1)), flat_m, flat_v, step, lr)
    np.maximum(sg, SIGMA_MIN, out=sg)
    lam[:, 0] += RHO * terms[:, oracle.T_VDEP]
    lam[:, 1] += RHO * terms[:, oracle.T_VRES]
    lam[:, 2] += RHO * terms[:, oracle.T_VREC]


def _oracle_setup(name, r):
    import oracle
    oracle.build()
    p, B, mu0, sg0 = workload(0, None, name)
    r = min(B, r)
    op = oracle.OracleProblem(p)
    ohp = oracle.hparams(tau=TAU, rho=RHO, alpha=ALPHA, w_res=W_RES, w_mem=W_MEM, terms=p.terms)
    mu = mu0[:, :r].astype(np.float64).copy()
    sg = sg0[:, :r].astype(np.float64).copy()
    lam = np.full((r, 3), LAMBDA0)
    mom = [np.zeros_like(mu) for _ in range(4)]
    return p, B, r, op, ohp, mu, sg, lam, mom


def cpu_sample(name, threads, budget):
    """The fp64 oracle, as it stands (OpenMP over restarts), on a bounded sample of
    the workload: whole iterations (loss, gradient, Adam, multipliers) of
    min(B, threads) restarts until `budget` seconds have passed (at least one, at most
    five).  Prints one JSON line."""
    p, B, r, op, ohp, mu, sg, lam, mom = _oracle_setup(name, threads)
    t0 = time.perf_counter()
    it = 0
    while True:
        it += 1
        _oracle_iteration(op, ohp, mu, sg, lam, mom, it, p.lr)
        el = time.perf_counter() - t0
        if el >= budget or it >= 5:
            break
    print(json.dumps({"value": r * it / el, "unit": UNIT, "cores": threads, "kind": "oracle",
                      "sample": f"{it} iteration(s) of {r} of the {B} restarts of {p.name}, fp64, unwindowed, "
                                f"{threads} thread(s), {el:.1f} s"}))


def cpu_sample_subprocess(name, threads, budget):
    """cpu_sample in a fresh interpreter with OMP_NUM_THREADS = threads."""
    env = dict(os.environ, OMP_NUM_THREADS=str(threads))
    cmd = [sys.executable, os.path.abspath(__file__), "--cpu-sample", name, "--threads", str(threads),
           "--budget", str(budget)]
    try:
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=3600)
        return json.loads(r.stdout.strip().splitlines()[-1])
    except Exception as e:  # the baseline is reported, never required
        return {"unavailable": f"{type(e).__name__}: {e}"[:200]}


def reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cores = os.cpu_count() or 1
    os.environ.setdefault("OMP_NUM_THREADS", str(cores))
    p, B, r, op, ohp, mu, sg, lam, mom = _oracle_setup(args.workload, cores)
    iters = args.iters or p.iters
    for w in range(args.warmup):
        _oracle_iteration(op, ohp, mu, sg, lam, mom, w + 1, p.lr)
    t0 = time.perf_counter()
    for k in range(args.steps):
        _oracle_iteration(op, ohp, mu, sg, lam, mom, args.warmup + k + 1, p.lr)
    el = time.perf_counter() - t0
    value = args.steps * r / el
    sample = f"1 iteration of {r} of the {B} restarts per step, fp64 oracle, unwindowed"
    headline = args.workload == HEADLINE
    print(json.dumps({"impl": "reference", "metric": METRIC if headline else
                      METRIC.replace("logic-network DAG, |V|=10k", p.name),
                      "value": value, "unit": UNIT, "n_gpus": 1,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                      "data": f"synthetic (seeded {p.name} DAG and initial means)",
                      "config": dict(describe(args.workload, p, B, iters, min(args.period, iters)), sample=sample),
                      "cpu_baseline": {"value": value, "unit": UNIT, "cores": int(os.environ["OMP_NUM_THREADS"]),
                                       "kind": "oracle", "sample": sample},
                      "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


if __name__ == "__main__":
    a = parse()
    if a.cpu_sample is not None:
        cpu_sample(a.cpu_sample, a.threads or (os.cpu_count() or 1), a.budget)
    elif a.phase_probe is not None:
        phase_probe(a)
    elif a.fused_probe is not None:
        fused_probe(a)
    elif a.impl == "reference":
        reference_arm(a)
    else:
        gpu_arm(a)
