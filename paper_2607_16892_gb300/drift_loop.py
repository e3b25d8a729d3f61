"""Host loop over drifting workloads: one reservation re-optimisation per iteration.

Each iteration redraws every class's output-length samples (lognormal medians
drift by +2% per iteration), uploads them from pinned host memory, sorts them,
takes the 64 fractile quantiles, evaluates the FP32 grid and reads back the
chosen reservation per (radius, class).  This is the shape of the outer loop of
the paper's BCD-DRO algorithm (Alg. 1) that calls the reservation evaluation once
per iteration; its other blocks (routing LP, caching rule, configuration
enumeration) are not part of this library.

The GPU time of an iteration runs from the host-to-device copy of its samples to
the end of its grid kernel (CUDA events on one stream).  While the GPU works on
iteration t the host draws iteration t+1.  One JSON line per iteration is written
to ``--out``; a run started with ``--resume`` skips the iterations already there
(each iteration's draws depend only on its index).

    python -m paper_2607_16892_gb300.drift_loop --iterations 50 --out drift.jsonl
"""

from __future__ import annotations

import argparse
import json
import os
import sys
import threading
import time

import numpy as np

from . import kvdro as kv


def _workload(t: int):
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    from synth import drift_loop_workload_k32_n1e6
    return drift_loop_workload_k32_n1e6(t)


def _done_iterations(path: str):
    done = set()
    if path and os.path.exists(path):
        for line in open(path):
            try:
                done.add(int(json.loads(line)["iteration"]))
            except (ValueError, KeyError):
                continue
    return done


def run(iterations: int = 50, out: str = "", resume: bool = False, device: int = 0, precision: int = kv.KVDRO_FP32,
        log=print):
    import torch

    dev = torch.device("cuda", device)
    torch.cuda.set_device(dev)
    done = _done_iterations(out) if resume else set()
    todo = [t for t in range(iterations) if t not in done]
    if not todo:
        return []
    ctx = kv.kvdro_create(device)
    stream = torch.cuda.current_stream(dev)
    records = []
    fh = open(out, "a") if out else None
    try:
        w = _workload(todo[0])
        M, E, K, R, NL, F = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam), len(w.fractiles)
        ft = torch.float32 if precision == kv.KVDRO_FP32 else torch.float64
        h_samples = [torch.empty(int(w.offsets[-1]), dtype=torch.int32).pin_memory() for _ in range(2)]
        d_samples = torch.empty(int(w.offsets[-1]), dtype=torch.int32, device=dev)
        quant = torch.empty((K, F), dtype=torch.int32, device=dev)
        r_idx = torch.empty((M, E, K), dtype=torch.int32, device=dev)
        min_cost = torch.empty((M, E, K), dtype=ft, device=dev)
        fhat = torch.empty((M, E, K), dtype=torch.float64, device=dev)
        h_samples[0].numpy()[:] = w.samples
        nxt = {}

        def draw(t, slot):
            nxt["w"] = _workload(t)
            h_samples[slot].numpy()[:] = nxt["w"].samples

        for n, t in enumerate(todo):
            slot = n % 2
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            ev[0].record(stream)
            d_samples.copy_(h_samples[slot], non_blocking=True)
            ev[1].record(stream)
            kv.kvdro_load_samples(ctx, K, w.offsets, d_samples, w.L, w.L_in, stream)
            kv.kvdro_quantiles(ctx, F, w.fractiles, quant, stream)
            ev[2].record(stream)
            kv.kvdro_eval_grid(ctx, precision, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, r_idx=r_idx,
                               min_cost=min_cost, fhat=fhat, stream=stream)
            ev[3].record(stream)
            drawer = None
            if n + 1 < len(todo):  # the host draws the next iteration while the GPU evaluates this one
                drawer = threading.Thread(target=draw, args=(todo[n + 1], 1 - slot))
                drawer.start()
            ev[3].synchronize()
            grid_ms = kv.kvdro_last_grid_ms(ctx)
            rec = {
                "iteration": t, "workload": w.name, "terms": w.terms(),
                "gpu_ms": ev[0].elapsed_time(ev[3]), "upload_ms": ev[0].elapsed_time(ev[1]),
                "sort_quantiles_ms": ev[1].elapsed_time(ev[2]), "eval_ms": ev[2].elapsed_time(ev[3]),
                "grid_kernel_ms": grid_ms, "terms_per_s": w.terms() / (grid_ms / 1e3),
                "r_star_eps0": w.r[r_idx[0, 0].cpu().numpy()].tolist(),
                "fhat_eps0": fhat[0, 0].cpu().numpy().round(6).tolist(),
                "median_quantile": quant[:, int(np.argmin(np.abs(w.fractiles - 0.5)))].cpu().numpy().tolist(),
            }
            records.append(rec)
            if fh:
                fh.write(json.dumps(rec) + "\n")
                fh.flush()
            log(f"iteration {t}: gpu {rec['gpu_ms']:.1f} ms (upload {rec['upload_ms']:.1f}, sort+quantiles "
                f"{rec['sort_quantiles_ms']:.1f}, eval {rec['eval_ms']:.1f}), {rec['terms_per_s']:.3e} terms/s")
            if drawer is not None:
                drawer.join()
                w = nxt["w"]
    finally:
        if fh:
            fh.close()
        kv.kvdro_destroy(ctx)
    return records


def main():
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--iterations", type=int, default=50)
    p.add_argument("--out", default="")
    p.add_argument("--resume", action="store_true")
    p.add_argument("--device", type=int, default=0)
    a = p.parse_args()
    t0 = time.perf_counter()
    recs = run(a.iterations, a.out, a.resume, a.device)
    if recs:
        g = [r["gpu_ms"] for r in recs]
        print(json.dumps({"iterations": len(recs), "gpu_ms_mean": float(np.mean(g)), "gpu_ms_max": float(np.max(g)),
                          "wall_s": time.perf_counter() - t0}))


if __name__ == "__main__":
    main()
