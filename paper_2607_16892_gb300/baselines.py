"""Baseline reservations and their costs next to the DRO reservation.

The paper compares its DRO reservation with fixed rules (Sec. 5.1 "Baselines": Max, Mean,
P90, P95 with block alignment, P99, SAA; Sec. 5.5: length prediction r = L_in + mu + k sigma
for k in {1, 2}) by their preemption/waste cost (Tables 2 and 4).  This module computes the
same rules from one class's samples and prices every rule with the library's exact dual
(`kvdro_eval_dual`): the empirical expected cost (radius 0) and the worst-case expected cost
over the 1-Wasserstein ball of each radius.  The SAA and DRO reservations are the argmins of
those costs over every integer reservation in [L_in, L_in + L].

Quantiles come from the GPU sort; the class mean and standard deviation used by the
length-prediction rule are taken on the host from the same samples.

    python -m paper_2607_16892_gb300.baselines --workload lognormal_k8_n1e5 --rho 2 10 100
"""

from __future__ import annotations

import argparse
import json
import math
import os
import sys
from typing import Dict, List, Sequence

import numpy as np

from . import kvdro as kv

RULES = ("max", "mean", "p90", "p95_block16", "p99", "lp_1sigma", "lp_2sigma")


def rule_reservations(w, quant: np.ndarray, block: int = 16) -> Dict[str, np.ndarray]:
    """r per class for each fixed rule (quant[k] = lower quantiles at 0.90, 0.95, 0.99)."""
    out = {}
    lo = w.L_in.astype(np.int64)
    hi = (w.L_in + w.L).astype(np.int64)
    mean = np.array([w.class_samples(k).mean() for k in range(w.K)])
    std = np.array([w.class_samples(k).std() for k in range(w.K)])
    clip = lambda v: np.clip(v, lo, hi).astype(np.int32)  # noqa: E731
    out["max"] = clip(hi)
    out["mean"] = clip(lo + np.ceil(mean))
    out["p90"] = clip(lo + quant[:, 0])
    out["p95_block16"] = clip(np.ceil((lo + quant[:, 1]) / block) * block)
    out["p99"] = clip(lo + quant[:, 2])
    out["lp_1sigma"] = clip(lo + np.ceil(mean + std))
    out["lp_2sigma"] = clip(lo + np.ceil(mean + 2 * std))
    return out


def compare(w, eps: Sequence[float], device: int = 0) -> List[dict]:
    """One record per (regime, class): every rule's r and cost at each radius, and the SAA and
    DRO reservations with theirs.  Costs are exact dual values (radius 0 = empirical cost)."""
    import torch

    eps = np.asarray(sorted(set([0.0] + list(eps))), np.float64)
    M, E, K = len(w.cp), len(eps), w.K
    dev = torch.device("cuda", device)
    ctx = kv.kvdro_create(device)
    try:
        kv.kvdro_load_samples(ctx, K, w.offsets, torch.from_numpy(w.samples).to(dev), w.L, w.L_in)
        quant = np.empty((K, 3), np.int32)
        kv.kvdro_quantiles(ctx, 3, [0.90, 0.95, 0.99], quant)
        rules = rule_reservations(w, quant)
        # every integer reservation valid for all classes
        grid = np.arange(int(w.L_in.max()), int((w.L_in + w.L).min()) + 1, dtype=np.int32)
        R = grid.size
        cost = np.empty((M, E, K, R), np.float64)
        r_idx = np.empty((M, E, K), np.int32)
        kv.kvdro_eval_dual(ctx, R, grid, E, eps, M, w.cp, w.cw, cost=cost, r_idx=r_idx)
    finally:
        kv.kvdro_destroy(ctx)
    recs = []
    for m in range(M):
        for k in range(K):
            rec = {"regime": m, "c_p": float(w.cp[m]), "c_w": float(w.cw[m]), "class": k,
                   "critical_fractile": float(w.cp[m] / (w.cp[m] + w.cw[m])), "eps": eps.tolist(), "rules": {}}
            for name in RULES:
                r = int(rules[name][k])
                i = r - int(grid[0])
                rec["rules"][name] = {"r": r, "cost": [float(cost[m, e, k, i]) if 0 <= i < R else None
                                                       for e in range(E)]}
            saa = int(r_idx[m, 0, k])
            rec["rules"]["saa"] = {"r": int(grid[saa]), "cost": [float(cost[m, e, k, saa]) for e in range(E)]}
            rec["dro"] = [{"eps": float(eps[e]), "r": int(grid[r_idx[m, e, k]]), "cost": float(cost[m, e, k, r_idx[m, e, k]])}
                          for e in range(E)]
            recs.append(rec)
    return recs


def main():
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    from synth import WORKLOADS, slice_workload

    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--workload", default="lognormal_k8_n1e5", choices=sorted(WORKLOADS))
    p.add_argument("--rho", type=float, nargs="*", default=[2.0, 10.0, 100.0], help="c_p / c_w regimes (c_w = 1)")
    p.add_argument("--eps", type=float, nargs="*", default=[10.0, 100.0], help="radii in tokens")
    a = p.parse_args()
    w = WORKLOADS[a.workload]()
    w = slice_workload(w, regimes=[0], name=w.name)
    w.cp = np.asarray(a.rho, np.float64)
    w.cw = np.ones_like(w.cp)
    for rec in compare(w, a.eps):
        print(json.dumps(rec))


if __name__ == "__main__":
    main()
