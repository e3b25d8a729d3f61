"""Run one grid pass of a workload through the C ABI (device memory from PyTorch).

Plumbing only: allocates device tensors for the inputs and outputs, calls the
library's entry points in order, and returns host copies.
"""

from __future__ import annotations

from typing import Dict, Iterable, Optional

import numpy as np

from .kvdro import (KVDRO_EXACT, KVDRO_FP32, KVDRO_FP64, kvdro_create, kvdro_destroy, kvdro_eval_grid, kvdro_load_samples,
                    kvdro_quantiles, kvdro_sorted_samples)

ALL_OUTPUTS = ("S", "cost", "lam_idx", "r_idx", "min_cost", "fhat", "quant", "sorted")


def run(w, precision: int = KVDRO_FP32, outputs: Iterable[str] = ALL_OUTPUTS, device: int = 0,
        host_outputs: bool = False, ctx=None) -> Dict[str, np.ndarray]:
    """Load ``w``'s samples, evaluate its grid and return the requested outputs as NumPy arrays.
    With ``host_outputs`` the library writes straight into host (NumPy) buffers."""
    import torch

    outputs = set(outputs)
    dev = torch.device("cuda", device)
    ft = torch.float32 if precision == KVDRO_FP32 else torch.float64
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    own = ctx is None
    if own:
        ctx = kvdro_create(device)
    try:
        samples = torch.from_numpy(np.ascontiguousarray(w.samples, np.int32)).to(dev)
        kvdro_load_samples(ctx, K, w.offsets, samples, w.L, w.L_in)

        def alloc(name, shape, dtype):
            if name not in outputs:
                return None
            if host_outputs:
                return np.empty(shape, dtype=np.dtype(str(dtype).replace("torch.", "")))
            return torch.empty(shape, dtype=dtype, device=dev)

        out = {
            "S": alloc("S", (M, K, R, NL), ft),
            "cost": alloc("cost", (M, E, K, R), ft),
            "lam_idx": alloc("lam_idx", (M, E, K, R), torch.int32),
            "r_idx": alloc("r_idx", (M, E, K), torch.int32),
            "min_cost": alloc("min_cost", (M, E, K), ft),
            "fhat": alloc("fhat", (M, E, K), torch.float64),
        }
        kvdro_eval_grid(ctx, precision, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw, S=out["S"], cost=out["cost"],
                        lam_idx=out["lam_idx"], r_idx=out["r_idx"], min_cost=out["min_cost"], fhat=out["fhat"])
        if "quant" in outputs:
            out["quant"] = alloc("quant", (K, len(w.fractiles)), torch.int32)
            kvdro_quantiles(ctx, len(w.fractiles), w.fractiles, out["quant"])
        if "sorted" in outputs:
            out["sorted"] = alloc("sorted", (int(w.offsets[-1]),), torch.int32)
            kvdro_sorted_samples(ctx, out["sorted"])
        torch.cuda.synchronize(dev)
        return {k: (v if isinstance(v, np.ndarray) else v.cpu().numpy()) for k, v in out.items() if v is not None}
    finally:
        if own:
            kvdro_destroy(ctx)
