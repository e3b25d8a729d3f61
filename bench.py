#!/usr/bin/env python3
"""Throughput of the Wasserstein-DRO reservation-cost path on one GB300 (or N replicas).

One step is one pass of the whole path over the regime-sweep workload, the largest of the
five workload configurations (8 classes x 200,000 samples; 2048 reservations x 64
multipliers x 16 radii x 1024 cost regimes c_p/c_w log-spaced over [1, 1000]; 2.15e14 cost
terms): load + range check + segmented sort of the samples, the 1024 critical-fractile
quantiles, the FP32 grid evaluation with its eps epilogue, and the argmin over r.  The
metric counts one cost term per (regime, class, r, lam, sample); eps does not multiply
per-sample work and is not counted.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]

Under torchrun each rank evaluates its own replica of the workload (independent
problems, no collective on the data path); the JSON line reports the sum of all
ranks' terms divided by the slowest rank's time.  ``--impl reference`` times the
CPU oracle on bounded samples of the same workload instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from synth import WORKLOADS, slice_workload  # noqa: E402

METRIC = "DRO cost terms/sec (class×r×λ×sample) on 1 GB300; % of FP32/HBM roofline"
UNIT = "terms/s"
DEFAULT_WORKLOAD = "regimes_k8_n2e5"
SM_MAX_MHZ_RECIPE = 2070.0
# Bound of the exact kernel's per-term work.  A term costs one instruction-lane on one of two
# pipes: packed f32x2 adds on the FMA pipe (128 FP32 lanes/clk/SM, two lane-operations per term:
# 64 terms/clk/SM) or an integer absolute-difference-and-add (sad) on the ALU pipe (64 lanes/clk/SM,
# one per term: 64 terms/clk/SM).  The kernel splits every warp's cells between the two, so at
# most 128 terms per clock per SM, which is also the issue limit (4 schedulers x 1 instruction per
# clock x 32 lanes, one instruction per term and lane).  Measured on this GB300: packed f32x2 adds
# alone 127.9 FP32 lane-ops/clk/SM, sad.s32 alone 63.4 terms/clk/SM.
FMA_TERMS_PER_CLK_PER_SM = 128.0 / 2.0
ALU_TERMS_PER_CLK_PER_SM = 64.0
TERMS_PER_CLK_PER_SM = FMA_TERMS_PER_CLK_PER_SM + ALU_TERMS_PER_CLK_PER_SM
# The per-term bound of the three-candidate supremum as written: two FMAs, two maxima and one add
# per term, 5 FP32 lane-operations on 128 FP32 lanes per clock per SM.
PAPER_FORM_LANE_OPS_PER_TERM = 5.0
# The FP32-arithmetic kernel's bound: per term one fused multiply-add and one add on the FP32 lanes
# (2 lane-operations of 128 per clock per SM) and one max on the ALU pipe alongside.
FP32_PHI_TERMS_PER_CLK_PER_SM = 128.0 / 2.0
# What the exact kernel evaluates per term: once a cell's exact integer threshold t is known
# (x >= t exactly when the excess kappa x + d is positive), the excess sum is
# kappa sum_{x >= t} x + d #{x >= t}, and the kernel streams sum_n |x_n - (t - 1)| to get it.
# That sum also has an O(1) closed form from the cumulative counts and sums the same context holds
# (the envelope mode returns the same S that way).
PER_TERM_OP = "|x - c| summed exactly per (cell, sample), c = t - 1 the cell's integer threshold; not the 3-candidate phi"
GRID_SOURCE = os.path.join(ROOT, "paper_2607_16892_gb300", "csrc", "grid.cu")
PROFILE = os.path.join(ROOT, "profiles", "k_grid_exact_regimes_k8_n2e5.md")
LAUNCHES_PER_STEP = 7  # histogram, scan totals, scan, expand, quantile gather, grid, argmin finalise
# FP64 pipe bound of the native FP64 mode: per term one DFMA (2.0 per clk per SM) plus one DADD and
# one max.f64 (1.7 per clk per SM each), measured on this GB300; nominal 1.25 TFLOP/s FP64.
FP64_TERMS_PER_CLK_PER_SM = 1.0 / (1.0 / 2.0 + 2.0 / 1.7)


def parse_args():
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(WORKLOADS),
                   help="workload configuration of a step (default: the largest, the regime sweep)")
    p.add_argument("--e2e-steps", type=int, default=2)
    p.add_argument("--cpu-seconds", type=float, default=10.0, help="target wall time of the CPU-baseline sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-phi-kernel", action="store_true",
                   help="skip the secondary figure of the per-term phi kernel (roofline.per_term_phi)")
    p.add_argument("--no-secondary", action="store_true",
                   help="skip the secondary figures (native FP64 on one regime, envelope and exact dual)")
    p.add_argument("--drift-iterations", type=int, default=3)
    p.add_argument("--case", default="",
                   help="WORKLOAD:MODE[:key=val,...], MODE in fp32|fp64|exact|envelope|dual|sort: time one kernel "
                        "path (--warmup untimed, --steps timed runs) and print one line per run.  Keys: L (support "
                        "declared for every class, e.g. 4194305 so FP32 requests take the FP32-arithmetic kernel), "
                        "nl (lam count, log-spaced over the workload's lam range), m (first m regimes), "
                        "rstride (every rstride-th r), out=all (write every output the contract step writes: "
                        "cost, lam index, r index, min cost, F-hat; default the r index only)")
    p.add_argument("--suite", action="store_true",
                   help="time every workload in each precision (one JSON line per case) instead of the contract line")
    p.add_argument("--cpu-suite", action="store_true",
                   help="time the CPU oracle (the reported baseline) on every workload, one line each")
    return p.parse_args()


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), int(os.environ.get("WORLD_SIZE", 1))


def workload_config(w, world):
    ratio = w.cp / w.cw
    return {
        "workload": w.name,
        "classes": int(w.K),
        "samples_per_class": int(w.N[0]),
        "r_points": int(len(w.r)),
        "lam_points": int(len(w.lam)),
        "eps_points": int(len(w.eps)),
        "regimes": int(len(w.cp)),
        "cost_ratio": float(ratio[0]) if len(ratio) == 1 else f"{len(ratio)} log-spaced in "
                                                              f"[{ratio.min():g}, {ratio.max():g}]",
        "support_L": int(w.L[0]),
        "fractiles": int(len(w.fractiles)),
        "terms_per_step_per_gpu": int(w.terms()),
        "step": "load+range check+segmented sort, quantiles, FP32 grid eval + eps epilogue + argmin over r",
        "outputs": "cost and lam index per (regime, eps, class, r); r index, min cost and F-hat per "
                   "(regime, eps, class); quantiles per (class, fractile)",
        "l2": "flushed between timed steps (256 MiB device write outside the timed events)",
        "parallelism": "single GPU" if world == 1 else f"{world} independent replicas (no data-path collective)",
    }


def phi_kernel_figure(kv, w, device, stream, sms, regimes=16, reps=2):
    """A secondary figure beside the headline: the FP32-arithmetic kernel, which evaluates phi's
    excess per term (one saturating fused multiply-add on the excess scaled by a power of two, whose
    clamp to [0, 1] is the max, and half a packed add per (cell, sample); FP32 sums folded into
    FP64), on the first `regimes` regimes of the same workload.  The same samples and
    grid with the support declared as 2^22 + 1, which is what routes FP32 requests to it; the
    supremum and the sum are unchanged (every sample and reservation lies in both supports)."""
    import torch

    sub = slice_workload(w, regimes=np.arange(min(regimes, len(w.cp))), name=w.name)
    L_big = np.full(sub.K, (1 << 22) + 1, np.int32)
    M, E, K, R, NL = len(sub.cp), len(sub.eps), sub.K, len(sub.r), len(sub.lam)
    ctx = kv.kvdro_create(device)
    try:
        d = torch.from_numpy(sub.samples).to(torch.device("cuda", device))
        kv.kvdro_load_samples(ctx, K, sub.offsets, d, L_big, sub.L_in, stream)
        r_idx = torch.empty((M, E, K), dtype=torch.int32, device=d.device)
        ms = []
        for i in range(reps + 1):
            kv.kvdro_eval_grid(ctx, kv.KVDRO_FP32, R, sub.r, NL, sub.lam, E, sub.eps, M, sub.cp, sub.cw,
                               r_idx=r_idx, stream=stream)
            if i:
                ms.append(kv.kvdro_last_grid_ms(ctx))
    finally:
        kv.kvdro_destroy(ctx)
    kernel_ms = statistics.mean(ms)
    achieved = sub.terms() / (kernel_ms / 1e3)
    peak_fp32 = sms * FP32_PHI_TERMS_PER_CLK_PER_SM * SM_MAX_MHZ_RECIPE * 1e6
    peak_paper = sms * 128.0 / PAPER_FORM_LANE_OPS_PER_TERM * SM_MAX_MHZ_RECIPE * 1e6
    return {"kernel": "k_grid<F32>: per term fma.rn.sat.f32 (max(kappa (x - eta) + W, 0) / S, S a power of two), "
                      "add.rn.f32x2 (sum)",
            "workload": f"{w.name}, first {M} of {len(w.cp)} regimes ({sub.terms():.4g} terms), support declared "
                        f"as 2^22 + 1", "kernel_ms_mean": kernel_ms, "achieved": achieved, "unit": UNIT,
            "frac": achieved / peak_fp32,
            "peak_basis": f"{sms} SMs x {FP32_PHI_TERMS_PER_CLK_PER_SM:.0f} terms/clk/SM (2 FP32 lane-ops per term "
                          f"on 128 lanes: the saturating FMA and the add) x {SM_MAX_MHZ_RECIPE:.0f} MHz",
            "frac_survey_basis": achieved / peak_paper}


def secondary_figures(kv, w, ctx, stream, sms, reps=2):
    """Beside the headline, outside its timed region, on the context that holds the workload's
    samples: the native FP64 per-term kernel on the first regime (a full FP64 pass takes about
    1000 s), and the two modes that are not per term -- the envelope sums and the exact dual over
    gamma >= 0 -- on the whole workload, in cells/s."""
    import torch

    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    dev = torch.device("cuda", torch.cuda.current_device())

    def timed(fn):
        ms = []
        for i in range(reps + 1):
            fn()
            if i:
                ms.append(kv.kvdro_last_grid_ms(ctx))
        return statistics.mean(ms)

    r1 = torch.empty((1, E, K), dtype=torch.int32, device=dev)
    fp64_ms = timed(lambda: kv.kvdro_eval_grid(ctx, kv.KVDRO_FP64, R, w.r, NL, w.lam, E, w.eps, 1, w.cp[:1],
                                               w.cw[:1], r_idx=r1, stream=stream))
    fp64_terms = R * NL * int(w.N.sum())
    fp64_rate = fp64_terms / (fp64_ms / 1e3)
    fp64_peak = sms * FP64_TERMS_PER_CLK_PER_SM * SM_MAX_MHZ_RECIPE * 1e6
    r_all = torch.empty((M, E, K), dtype=torch.int32, device=dev)
    env_ms = timed(lambda: kv.kvdro_eval_grid(ctx, kv.KVDRO_ENVELOPE, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw,
                                              r_idx=r_all, stream=stream))
    dual_ms = timed(lambda: kv.kvdro_eval_dual(ctx, R, w.r, E, w.eps, M, w.cp, w.cw, r_idx=r_all, stream=stream))
    return {"fp64_per_term": {"kernel": "k_grid<F64>: per term one DFMA, one max.f64, one DADD",
                              "workload": f"{w.name}, first regime ({fp64_terms:.4g} terms)", "kernel_ms": fp64_ms,
                              "achieved": fp64_rate, "unit": UNIT, "peak": fp64_peak, "frac": fp64_rate / fp64_peak,
                              "peak_basis": f"{sms} SMs x {FP64_TERMS_PER_CLK_PER_SM:.3f} terms/clk/SM (measured FP64 "
                                            f"pipe rates: 2.0 DFMA, 1.7 DADD / max.f64 per clk per SM) x "
                                            f"{SM_MAX_MHZ_RECIPE:.0f} MHz"},
            "envelope": {"what": "O(1) per cell from cumulative counts and sums; not per term",
                         "cells": M * K * R * NL, "kernel_ms": env_ms, "cells_per_s": M * K * R * NL / (env_ms / 1e3)},
            "exact_dual": {"what": "min over gamma >= 0 by bisection, O(1) per probe; not per term",
                           "cells": M * E * K * R, "kernel_ms": dual_ms, "cells_per_s": M * E * K * R / (dual_ms / 1e3)}}


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the architecture)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        fields = {ln.split(":", 1)[0].strip(): ln.split(":", 1)[1].strip() for ln in out.splitlines() if ":" in ln}
        name = fields.get("Model name", "")
        if name and name != "-":
            vendor = fields.get("Vendor ID", "")
            return f"{vendor} {name}".strip() if vendor and vendor not in name else name
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu part")):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.machine()


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi clock and throttle-reason samples during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id: str):
        self.proc = None
        self.path = None
        self.gpu_id = gpu_id

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="kvdro_clocks_", suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, smax, reasons = [], [], set()
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for name, val in zip(self.REASONS, f[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ helpers

def reduce_max(value: float, device=None) -> float:
    """Maximum of a per-rank scalar over all ranks (identity when not distributed)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(terms_per_rank_step: int, steps: int, world: int, slowest_s: float) -> float:
    """Whole-job throughput: every rank's terms over the slowest rank's time."""
    return terms_per_rank_step * steps * world / slowest_s


def profile_figures():
    """DRAM bytes per grid-kernel launch and warp instructions per term-lane from the committed
    ncu summary, if it was taken on the current kernel source (else None for both)."""
    try:
        text = open(PROFILE).read()
        src_hash = hashlib.sha256(open(GRID_SOURCE, "rb").read()).hexdigest()
    except OSError:
        return None, None
    m_hash = re.search(r"grid_cu_sha256:\s*([0-9a-f]{64})", text)
    if not m_hash or m_hash.group(1) != src_hash:
        return None, None
    m_traf = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    m_inst = re.search(r"inst_per_term:\s*([0-9.eE+]+)", text)
    return (float(m_traf.group(1)) if m_traf else None), (float(m_inst.group(1)) if m_inst else None)


def oracle_rows(w, rows: int):
    """Cells of `rows` (regime, r) rows strided over the workload's M x R rows, each with every
    class and every lam value: the bounded sample the CPU oracle is timed on."""
    M, K, R, NL = len(w.cp), w.K, len(w.r), len(w.lam)
    pick = np.linspace(0, M * R - 1, rows).round().astype(np.int64)
    m, ri = np.divmod(pick, R)
    mm = np.repeat(m, K * NL)
    kk = np.tile(np.repeat(np.arange(K), NL), rows)
    rr = np.repeat(ri, K * NL)
    ll = np.tile(np.arange(NL), rows * K)
    return (mm.astype(np.int32), kk, rr, ll), int(rows * NL * int(w.N.sum()))


def cpu_baseline(w, seconds: float):
    """The CPU oracle (direct per-term FP64 evaluation, all host cores) on a bounded sample of the
    workload: strided (regime, r) rows with every class, the full lam grid and all samples."""
    from oracle import oracle as O

    threads = O.default_threads()
    K, NL = w.K, len(w.lam)
    cal, _ = oracle_rows(w, 1)
    t0 = time.perf_counter()
    O.eval_cells(w, *cal, threads=threads)
    t_cal = max(time.perf_counter() - t0, 1e-3)
    rows = int(max(1, min(len(w.cp) * len(w.r), seconds / t_cal)))
    cells, terms = oracle_rows(w, rows)
    t0 = time.perf_counter()
    O.eval_cells(w, *cells, threads=threads)
    dt = time.perf_counter() - t0
    return {"value": terms / dt, "unit": UNIT, "cores": threads, "cpu_model": cpu_model(), "kind": "oracle",
            "sample": f"{rows} strided (regime, r) rows x {NL} lam x {K} classes x {int(w.N[0])} samples = "
                      f"{terms:.3e} terms, direct per-term FP64 oracle, {dt:.2f} s wall"}, dt


# ------------------------------------------------------------------ our implementation

def run_ours(args):
    import torch

    rank, local_rank, world = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group(backend="nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    from paper_2607_16892_gb300 import kvdro as kv

    w = WORKLOADS[args.workload]()
    M, E, K, R, NL, F = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam), len(w.fractiles)
    terms = w.terms()
    ctx = kv.kvdro_create(local_rank)
    stream = torch.cuda.current_stream(dev)
    d_samples = torch.from_numpy(w.samples).to(dev)
    out = {
        "cost": torch.empty((M, E, K, R), dtype=torch.float32, device=dev),
        "lam_idx": torch.empty((M, E, K, R), dtype=torch.int32, device=dev),
        "r_idx": torch.empty((M, E, K), dtype=torch.int32, device=dev),
        "min_cost": torch.empty((M, E, K), dtype=torch.float32, device=dev),
        "fhat": torch.empty((M, E, K), dtype=torch.float64, device=dev),
    }
    quant = torch.empty((K, F), dtype=torch.int32, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def step(samples, outs, q):
        kv.kvdro_load_samples(ctx, K, w.offsets, samples, w.L, w.L_in, stream)
        kv.kvdro_quantiles(ctx, F, w.fractiles, q, stream)
        kv.kvdro_eval_grid(ctx, kv.KVDRO_FP32, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, cost=outs["cost"],
                           lam_idx=outs["lam_idx"], r_idx=outs["r_idx"], min_cost=outs["min_cost"],
                           fhat=outs["fhat"], stream=stream)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    for _ in range(args.warmup):
        step(d_samples, out, quant)
    torch.cuda.synchronize(dev)

    props = torch.cuda.get_device_properties(dev)
    gpu_id = str(getattr(props, "uuid", local_rank))
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) == 36:
        gpu_id = "GPU-" + gpu_id
    sampler = ClockSampler(gpu_id)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    grid_ms = []
    barrier()
    torch.cuda.synchronize(dev)
    sampler.start()
    wall0 = time.perf_counter()
    for i in range(args.steps):
        flush.zero_()  # evict the previous step's data from L2, outside the timed events
        starts[i].record(stream)
        step(d_samples, out, quant)
        ends[i].record(stream)
        grid_ms.append(kv.kvdro_last_grid_ms(ctx))
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - wall0
    barrier()
    clocks = sampler.stop()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    total_s = reduce_max(sum(step_ms) / 1e3, dev)
    value = weak_scaling_value(terms, args.steps, world, total_s)

    # roofline of the grid kernel (this rank's launches)
    kernel_ms = statistics.mean(grid_ms)
    achieved = terms / (kernel_ms / 1e3)
    sms = props.multi_processor_count
    peak = sms * TERMS_PER_CLK_PER_SM * SM_MAX_MHZ_RECIPE * 1e6
    peak_paper = sms * 128.0 / PAPER_FORM_LANE_OPS_PER_TERM * SM_MAX_MHZ_RECIPE * 1e6
    traffic, inst_per_term = profile_figures()
    roofline = {"bound": "alu", "achieved": achieved, "peak": peak, "unit": UNIT, "frac": achieved / peak,
                "traffic": traffic, "kernel": "k_grid<EXACT> (FP32 outputs)",
                "kernel_ms_mean": kernel_ms, "per_term_op": PER_TERM_OP,
                "peak_basis": f"{sms} SMs x ({FMA_TERMS_PER_CLK_PER_SM:.0f} terms/clk/SM on packed "
                              f"FP32 adds + {ALU_TERMS_PER_CLK_PER_SM:.0f} on integer sad) x {SM_MAX_MHZ_RECIPE:.0f} MHz",
                "frac_survey_basis": achieved / peak_paper,
                "survey_basis": f"{sms} SMs x 128 FP32 lanes / {PAPER_FORM_LANE_OPS_PER_TERM:.0f} lane-ops per term of "
                                f"the 3-candidate phi (2 FMA, 2 max, 1 add) x {SM_MAX_MHZ_RECIPE:.0f} MHz = "
                                f"{peak_paper:.4g} terms/s; the kernel does not do that work per term",
                "inst_per_term": inst_per_term}
    if clocks.get("sm_mhz"):
        roofline["frac_at_sampled_clock"] = achieved / (peak * clocks["sm_mhz"] / SM_MAX_MHZ_RECIPE)
    if not args.no_phi_kernel:
        roofline["per_term_phi"] = phi_kernel_figure(kv, w, local_rank, stream, sms)
    secondary = None if args.no_secondary else secondary_figures(kv, w, ctx, stream, sms)

    # end to end through the C ABI with host buffers: pinned host samples in, host results out
    h_samples = torch.from_numpy(w.samples).pin_memory()
    h_out = {k: torch.empty(v.shape, dtype=v.dtype).pin_memory() for k, v in out.items()}
    h_quant = torch.empty(quant.shape, dtype=quant.dtype).pin_memory()
    step(h_samples, h_out, h_quant)
    torch.cuda.synchronize(dev)
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.e2e_steps):
        step(h_samples, h_out, h_quant)
    torch.cuda.synchronize(dev)
    e2e_s = reduce_max(time.perf_counter() - t0, dev)
    small_in = sum(a.nbytes for a in (w.offsets, w.L, w.L_in, w.r, w.lam, w.eps, w.cp, w.cw, w.fractiles))
    h2d = int(h_samples.numel() * 4 + small_in)
    d2h = int(sum(v.numel() * v.element_size() for v in h_out.values()) + h_quant.numel() * 4)
    e2e = {"value": weak_scaling_value(terms, args.e2e_steps, world, e2e_s), "unit": UNIT, "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu, _ = cpu_baseline(w, args.cpu_seconds)

    kv.kvdro_destroy(ctx)
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * total_s / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": workload_config(w, world), "roofline": roofline, "secondary": secondary,
            "cpu_baseline": cpu, "e2e": e2e,
            "clocks": {k: clocks[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
            "gpu_launches": LAUNCHES_PER_STEP * args.steps,
            "wall_s_timed_region": wall,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


# ------------------------------------------------------------------ reference arm (the CPU oracle)

def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return
    w = WORKLOADS[args.workload]()
    from oracle import oracle as O

    threads = O.default_threads()
    K, NL = w.K, len(w.lam)
    rows = 2  # per step: 2 strided (regime, r) rows x all lam x all classes x all samples
    cells, step_terms = oracle_rows(w, rows)
    for _ in range(args.warmup):
        O.eval_cells(w, *cells, threads=threads)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        O.eval_cells(w, *cells, threads=threads)
    dt = time.perf_counter() - t0
    value = step_terms * args.steps / dt
    sample = (f"per step {rows} strided (regime, r) rows x {NL} lam x {K} classes x {int(w.N[0])} samples = "
              f"{step_terms:.3e} terms, direct per-term FP64 oracle")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w, world),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "cpu_model": cpu_model(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_suite(args):
    """Grid throughput on every workload and precision (device-resident samples, kernel time from
    the library's CUDA events); plus a few iterations of the drifting-workload loop."""
    import torch

    from paper_2607_16892_gb300 import kvdro as kv
    from paper_2607_16892_gb300.drift_loop import run as drift_run
    from synth import WORKLOADS

    dev = torch.device("cuda", 0)
    props = torch.cuda.get_device_properties(dev)
    peak32 = props.multi_processor_count * TERMS_PER_CLK_PER_SM * SM_MAX_MHZ_RECIPE * 1e6
    peak64 = props.multi_processor_count * FP64_TERMS_PER_CLK_PER_SM * SM_MAX_MHZ_RECIPE * 1e6
    names = {kv.KVDRO_FP32: "fp32", kv.KVDRO_FP64: "fp64", kv.KVDRO_EXACT: "exact"}
    # bring the clocks up before the first measurement: a few seconds of the FP32 grid kernel
    warm = WORKLOADS["lognormal_k8_n1e5"]()
    wctx = kv.kvdro_create(0)
    kv.kvdro_load_samples(wctx, warm.K, warm.offsets, torch.from_numpy(warm.samples).to(dev), warm.L, warm.L_in)
    for _ in range(60):
        kv.kvdro_eval_grid(wctx, kv.KVDRO_FP32, len(warm.r), warm.r, len(warm.lam), warm.lam, len(warm.eps), warm.eps,
                           1, warm.cp, warm.cw)
    kv.kvdro_sync(wctx)
    kv.kvdro_destroy(wctx)
    cases = [("lognormal_k3_n1e3", [kv.KVDRO_FP64, kv.KVDRO_EXACT, kv.KVDRO_FP32]),
             ("lognormal_k8_n1e5", [kv.KVDRO_FP32, kv.KVDRO_EXACT, kv.KVDRO_FP64]),
             ("heavytail_k16_n1e6", [kv.KVDRO_FP32, kv.KVDRO_EXACT]),
             ("regimes_k8_n2e5", [kv.KVDRO_FP32, kv.KVDRO_EXACT])]
    for name, precs in cases:
        w = WORKLOADS[name]()
        ctx = kv.kvdro_create(0)
        d = torch.from_numpy(w.samples).to(dev)
        M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
        t0 = time.perf_counter()
        kv.kvdro_load_samples(ctx, K, w.offsets, d, w.L, w.L_in)
        load_ms = (time.perf_counter() - t0) * 1e3
        for prec in precs:
            r_idx = torch.empty((M, E, K), dtype=torch.int32, device=dev)
            reps = 1 if (prec == kv.KVDRO_FP64 or w.terms() > 1e13) else 3
            kv.kvdro_eval_grid(ctx, prec, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, r_idx=r_idx)
            ms = []
            for _ in range(reps):
                kv.kvdro_eval_grid(ctx, prec, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, r_idx=r_idx)
                ms.append(kv.kvdro_last_grid_ms(ctx))
            grid_ms = float(np.median(ms))
            rate = w.terms() / (grid_ms / 1e3)
            peak = peak64 if prec == kv.KVDRO_FP64 else peak32
            print(json.dumps({"suite": True, "workload": w.name, "precision": names[prec], "terms": w.terms(),
                              "grid_ms": grid_ms, "terms_per_s": rate, "peak": peak, "frac": rate / peak,
                              "load_sort_ms_wall": load_ms}), flush=True)
        # not per term: the envelope mode (cells/s) and the exact dual over gamma ((m, e, k, r) cells/s)
        for mode, label in ((kv.KVDRO_ENVELOPE, "envelope"), ("dual", "dual")):
            r_idx = torch.empty((M, E, K), dtype=torch.int32, device=dev)
            ms = []
            for _ in range(3):
                if mode == "dual":
                    kv.kvdro_eval_dual(ctx, R, w.r, E, w.eps, M, w.cp, w.cw, r_idx=r_idx)
                else:
                    kv.kvdro_eval_grid(ctx, mode, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, r_idx=r_idx)
                ms.append(kv.kvdro_last_grid_ms(ctx))
            grid_ms = float(np.median(ms[1:]))
            cells = M * K * R * NL if mode != "dual" else M * E * K * R
            print(json.dumps({"suite": True, "workload": w.name, "mode": label, "cells": cells, "grid_ms": grid_ms,
                              "cells_per_s": cells / (grid_ms / 1e3)}), flush=True)
        kv.kvdro_destroy(ctx)
    recs = drift_run(iterations=args.drift_iterations, log=lambda *_: None)
    for r in recs:
        print(json.dumps({"suite": True, **{k: r[k] for k in ("workload", "iteration", "terms", "gpu_ms", "upload_ms",
                                                                "sort_quantiles_ms", "eval_ms", "grid_kernel_ms",
                                                                "terms_per_s")}}), flush=True)


def run_cpu_suite(args):
    """The CPU oracle -- the reported baseline, never tuned -- on every workload: the direct
    per-term FP64 evaluation on all host cores and on one (the 3-class workload in full, 16 strided
    (regime, class, r) rows of the others, every lam and sample), the envelope regrouping
    (cells/s; a different algorithm), and its quantiles (a sort of every class)."""
    from oracle import oracle as O
    from synth import WORKLOADS

    threads = O.default_threads()
    for name in ("lognormal_k3_n1e3", "lognormal_k8_n1e5", "heavytail_k16_n1e6", "regimes_k8_n2e5", "drift_k32_n1e6"):
        w = WORKLOADS[name]()
        M, K, R, NL = len(w.cp), w.K, len(w.r), len(w.lam)
        rows_all = M * K * R
        full = name == "lognormal_k3_n1e3"
        n_rows = rows_all if full else 16
        pick = np.arange(rows_all) if full else np.linspace(0, rows_all - 1, n_rows).round().astype(np.int64)

        def cells(rows):
            m, rest = np.divmod(rows, K * R)
            k, r = np.divmod(rest, R)
            mm, ll = np.repeat(m, NL), np.tile(np.arange(NL), rows.size)
            return mm.astype(np.int32), np.repeat(k, NL), np.repeat(r, NL), ll

        def terms(rows):
            _, rest = np.divmod(rows, K * R)
            return int(sum(int(w.N[k]) for k in rest // R) * NL)

        t0 = time.perf_counter()
        O.eval_cells(w, *cells(pick), threads=threads)
        t_all = time.perf_counter() - t0
        one = pick[: max(1, min(pick.size, 2 if not full else pick.size))]
        t0 = time.perf_counter()
        O.eval_cells(w, *cells(one), threads=1)
        t_one = time.perf_counter() - t0
        we = w if M <= 16 else slice_workload(w, regimes=list(range(0, M, M // 16)), name=w.name)
        t0 = time.perf_counter()
        O.envelope_grid(we, threads=threads)
        t_env = time.perf_counter() - t0
        env_cells = len(we.cp) * K * R * NL
        t0 = time.perf_counter()
        O.quantiles(w, w.fractiles)
        t_sort = time.perf_counter() - t0
        print(json.dumps({"cpu_suite": True, "workload": w.name, "kind": "oracle",
                          "direct_terms_per_s": terms(pick) / t_all, "direct_cores": threads,
                          "direct_sample": f"{pick.size} (regime, class, r) rows x {NL} lam x all samples",
                          "direct_terms_per_s_one_core": terms(one) / t_one,
                          "envelope_cells_per_s": env_cells / t_env, "envelope_cells": env_cells,
                          "sort_quantiles_s": t_sort, "samples": int(w.N.sum())}), flush=True)


def case_options(spec: str) -> dict:
    parts = spec.split(":")
    return dict(kv.split("=") for kv in parts[2].split(",")) if len(parts) > 2 and parts[2] else {}


def case_workload(spec: str):
    """The workload of a --case spec WORKLOAD:MODE[:key=val,...] and its mode (see --case)."""
    parts = spec.split(":")
    name, mode = parts[0], parts[1]
    opts = case_options(spec)
    w = WORKLOADS[name]()
    if "m" in opts or "rstride" in opts:
        regimes = np.arange(int(opts.get("m", len(w.cp))))
        r_index = np.arange(0, len(w.r), int(opts.get("rstride", 1)))
        w = slice_workload(w, regimes=regimes, r_index=r_index, name=w.name)
    if "nl" in opts:
        w.lam = np.logspace(np.log10(w.lam[0]), np.log10(w.lam[-1]), int(opts["nl"]))
    if "L" in opts:  # a larger declared support: same samples, same grid
        w.L = np.full(w.K, int(opts["L"]), np.int32)
    return w, mode


def run_case(args):
    """One workload through one path, for profiling: load + sort, then the chosen evaluation."""
    import torch

    from paper_2607_16892_gb300 import kvdro as kv

    w, mode = case_workload(args.case)
    dev = torch.device("cuda", 0)
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    ctx = kv.kvdro_create(0)
    d = torch.from_numpy(w.samples).to(dev)
    r_idx = torch.empty((M, E, K), dtype=torch.int32, device=dev)
    prec = {"fp32": kv.KVDRO_FP32, "fp64": kv.KVDRO_FP64, "exact": kv.KVDRO_EXACT, "envelope": kv.KVDRO_ENVELOPE}
    outs = {}
    if case_options(args.case).get("out") == "all" and mode not in ("dual", "sort"):
        ft = torch.float32 if mode == "fp32" else torch.float64
        outs = {"cost": torch.empty((M, E, K, R), dtype=ft, device=dev),
                "lam_idx": torch.empty((M, E, K, R), dtype=torch.int32, device=dev),
                "min_cost": torch.empty((M, E, K), dtype=ft, device=dev),
                "fhat": torch.empty((M, E, K), dtype=torch.float64, device=dev)}
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        kv.kvdro_load_samples(ctx, K, w.offsets, d, w.L, w.L_in)
        if mode == "dual":
            kv.kvdro_eval_dual(ctx, R, w.r, E, w.eps, M, w.cp, w.cw, r_idx=r_idx)
        elif mode != "sort":
            kv.kvdro_eval_grid(ctx, prec[mode], R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, r_idx=r_idx, **outs)
        torch.cuda.synchronize(dev)
        line = {"case": args.case, "run": i, "timed": i >= args.warmup, "wall_ms": 1e3 * (time.perf_counter() - t0)}
        if mode not in ("sort", "dual", "envelope"):
            line["terms"] = w.terms()
        if mode != "sort":
            line["kernel_ms"] = kv.kvdro_last_grid_ms(ctx)
            if "terms" in line:
                line["terms_per_s"] = w.terms() / (line["kernel_ms"] / 1e3)
        print(json.dumps(line), flush=True)
    kv.kvdro_destroy(ctx)


def main():
    args = parse_args()
    if args.case:
        run_case(args)
        return
    if args.cpu_suite:
        run_cpu_suite(args)
        return
    if args.suite:
        run_suite(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
