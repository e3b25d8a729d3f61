"""Comparison rules between the CUDA path and the oracle (test infrastructure).

Tolerances are those the workloads are quoted with: 1e-9 relative for the FP64
path, 1e-5 relative for the FP32 path.  Integer outputs (sorted samples,
quantiles) must match bit for bit.  An argmin index must equal the oracle's
wherever the oracle's runner-up is more than the tolerance away; otherwise the
GPU's choice must have an oracle value within the tolerance of the minimum
(several indices are then correct).
"""

from __future__ import annotations

import numpy as np

RTOL = {"fp32": 1e-5, "fp64": 1e-9, "exact": 1e-9}


def rel_close(gpu, ref, rtol, what="", floor=0.0):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    err = np.abs(gpu - ref)
    bound = rtol * np.maximum(np.abs(ref), floor)
    bad = ~(err <= bound)
    if bad.any():
        i = np.unravel_index(np.argmax(np.where(bad, err / np.maximum(bound, 1e-300), 0)), ref.shape)
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside rtol {rtol}; worst at {i}: "
                             f"gpu {gpu[i]!r} ref {ref[i]!r} rel {err[i] / max(abs(ref[i]), 1e-300):.3e}")
    return float(np.max(err / np.maximum(np.abs(ref), 1e-300))) if ref.size else 0.0


def check_argmin(gpu_idx, ref_vals, rtol, what=""):
    """gpu_idx[...] chooses along the last axis of ref_vals[..., n] (vectorised rule above)."""
    gpu_idx = np.asarray(gpu_idx).reshape(-1).astype(np.int64)
    v = np.asarray(ref_vals, np.float64).reshape(-1, np.shape(ref_vals)[-1])
    assert gpu_idx.size == v.shape[0], what
    assert np.all((gpu_idx >= 0) & (gpu_idx < v.shape[1])), f"{what}: index out of range"
    b = np.argmin(v, axis=1)
    b1 = v[np.arange(v.shape[0]), b]
    tol = rtol * np.maximum(np.abs(b1), 1e-300)
    if v.shape[1] > 1:
        w = v.copy()
        w[np.arange(v.shape[0]), b] = np.inf
        b2 = w.min(axis=1)
    else:
        b2 = np.full_like(b1, np.inf)
    clear = (b2 - b1) > tol
    bad_exact = clear & (gpu_idx != b)
    assert not bad_exact.any(), (f"{what}: {bad_exact.sum()} indices differ where the runner-up gap exceeds tol; "
                                 f"first row {np.argmax(bad_exact)}")
    chosen = v[np.arange(v.shape[0]), gpu_idx]
    bad_tie = ~clear & (chosen > b1 + tol)
    assert not bad_tie.any(), f"{what}: {bad_tie.sum()} near-tie choices outside tol"
    return int(clear.sum())


def oracle_from_S(w, S):
    """The oracle's reductions of a given S grid (from the direct or the envelope evaluator)."""
    from oracle import oracle as O
    cost, lam_idx = O.eps_epilogue(S, w.lam, w.eps)
    r_idx, min_cost = O.argmin_r(cost)
    return dict(S=S, cost=cost, lam_idx=lam_idx, r_idx=r_idx, min_cost=min_cost, fhat=O.fhat_at(w, r_idx),
                quant=O.quantiles(w, w.fractiles))


def compare_full(w, gpu, ora, prec: str, check_S=True):
    """Every output of one grid pass against the oracle's solve()."""
    rtol = RTOL[prec]
    report = {}
    if check_S and "S" in gpu:
        report["S_max_rel"] = rel_close(gpu["S"], ora["S"], rtol, "S")
    if "cost" in gpu:
        report["cost_max_rel"] = rel_close(gpu["cost"], ora["cost"], rtol, "cost")
    if "lam_idx" in gpu:
        n_exact = 0
        for e, ep in enumerate(w.eps):
            obj = w.lam[None, None, None, :] * ep + ora["S"]   # [m, k, r, j]
            n_exact += check_argmin(gpu["lam_idx"][:, e], obj, rtol, f"lam_idx[eps {e}]")
        report["lam_idx_exact"] = n_exact
    if "r_idx" in gpu:
        report["r_idx_exact"] = check_argmin(gpu["r_idx"], ora["cost"], rtol, "r_idx")
    if "min_cost" in gpu:
        report["min_cost_max_rel"] = rel_close(gpu["min_cost"], ora["min_cost"], rtol, "min_cost")
    if "fhat" in gpu:
        # empirical CDF at the GPU's own r*, exactly
        for k in range(w.K):
            xs = np.sort(w.class_samples(k))
            eta = w.r[gpu["r_idx"][:, :, k]].astype(np.int64) - int(w.L_in[k])
            want = np.searchsorted(xs, eta, side="right") / xs.size
            assert np.array_equal(gpu["fhat"][:, :, k], want), "fhat"
    if "quant" in gpu:
        assert np.array_equal(gpu["quant"], ora["quant"]), "quantiles differ"
    if "sorted" in gpu:
        want = np.concatenate([np.sort(w.class_samples(k)) for k in range(w.K)])
        assert np.array_equal(gpu["sorted"], want), "sorted samples differ"
    return report
