"""CPU oracle for the Wasserstein-DRO reservation-cost grid (TEST INFRASTRUCTURE).

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg
may import this module.  It is the slow, plain, FP64 statement of what the CUDA
library computes, written from the paper (Appendix A, Prop. "Worst-Case
Expectation Reformulation"; Prop. "Critical Fractile Structure"), and it shares
no code with the library.

Layers:
  * ``kvdro_oracle.c`` (built here with gcc, loaded with ctypes): Q, phi, the
    per-cell sample mean S (direct, sequential FP64 sums), and the envelope
    regrouping of the same sum from exact cumulative counts.
  * this file (NumPy, FP64): the eps epilogue ``cost = min_j(lam_j eps + S_j)``,
    the argmin over r, the empirical CDF at the chosen r, and quantiles.

Readings where the paper is silent (ties, quantile convention) are stated in
each function's docstring.  Parity status: every function here is pinned by
the ``tests/test_oracle_*.py`` checks (brute force, LP duality, closed forms,
invariants, a hand-worked example); none is unpinned.
"""

from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from typing import Dict, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvdro_oracle.c")
_LIB = os.path.join(_HERE, "_build", "libkvdro_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle's C part with gcc (strict IEEE double: no FMA contraction)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-pthread",
               _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            d, i32, i64 = ctypes.c_double, ctypes.c_int32, ctypes.c_int64
            P = ctypes.c_void_p
            lib.kvo_Q.restype = d
            lib.kvo_Q.argtypes = [d, d, d, d]
            lib.kvo_phi.restype = d
            lib.kvo_phi.argtypes = [d, d, d, d, d, d]
            lib.kvo_mean_sup.restype = d
            lib.kvo_mean_sup.argtypes = [P, i64, d, d, d, d, d]
            lib.kvo_eval_cells.restype = ctypes.c_int
            lib.kvo_eval_cells.argtypes = [P, P, P, P, P, P, P, P, i64, P, P, P, P, P, ctypes.c_int]
            lib.kvo_cumulative.restype = ctypes.c_int
            lib.kvo_cumulative.argtypes = [P, i64, i32, P, P]
            lib.kvo_envelope_sum.restype = d
            lib.kvo_envelope_sum.argtypes = [P, P, i32, d, d, d, d]
            lib.kvo_exact_dual.restype = None
            lib.kvo_exact_dual.argtypes = [P, P, i32, i64, P, i64, d, d, d, d, P, P]
            lib.kvo_exact_dual_grid.restype = ctypes.c_int
            lib.kvo_exact_dual_grid.argtypes = [P, P, i64, P, P, P, P, P, P, P, P, P, i32, i32, i32, i32, P, P,
                                                ctypes.c_int]
            lib.kvo_envelope_grid.restype = ctypes.c_int
            lib.kvo_envelope_grid.argtypes = [P, P, i64, P, P, P, P, P, P, P, i32, i32, i32, i32, P, ctypes.c_int]
            _lib = lib
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


# ---------------------------------------------------------------- scalar pieces

def Q(eta: float, xi: float, cp: float, cw: float) -> float:
    """Stochastic reservation cost c_p (xi - eta)^+ + c_w (eta - xi)^+ (Sec. 2.3, App. A Step 1)."""
    return _load().kvo_Q(float(eta), float(xi), float(cp), float(cw))


def phi(x: float, eta: float, lam: float, cp: float, cw: float, L: float) -> float:
    """Closed-form pointwise sup over xi in [0, L] of Q(eta, xi) - lam |xi - x| (App. A Step 4)."""
    return _load().kvo_phi(float(x), float(eta), float(lam), float(cp), float(cw), float(L))


def mean_sup(x: np.ndarray, eta: float, lam: float, cp: float, cw: float, L: float) -> float:
    """(1/N) sum_n phi(x_n) with a sequential FP64 sum (App. A Step 3)."""
    x = np.ascontiguousarray(x, dtype=np.int32)
    return _load().kvo_mean_sup(_p(x), x.size, float(eta), float(lam), float(cp), float(cw), float(L))


# ---------------------------------------------------------------- grid evaluation

def _arrays(w):
    return dict(samples=np.ascontiguousarray(w.samples, np.int32),
                offsets=np.ascontiguousarray(w.offsets, np.int64),
                L=np.ascontiguousarray(w.L, np.int32),
                L_in=np.ascontiguousarray(w.L_in, np.int32),
                r=np.ascontiguousarray(w.r, np.int32),
                lam=np.ascontiguousarray(w.lam, np.float64),
                cp=np.ascontiguousarray(w.cp, np.float64),
                cw=np.ascontiguousarray(w.cw, np.float64))


def eval_cells(w, cell_m, cell_k, cell_r, cell_l, threads: Optional[int] = None) -> np.ndarray:
    """S(eta, lam) for a list of cells (regime index, class index, r index, lam index),
    each evaluated by the direct sample mean."""
    a = _arrays(w)
    cm = np.ascontiguousarray(cell_m, np.int32)
    ck = np.ascontiguousarray(cell_k, np.int32)
    cr = np.ascontiguousarray(cell_r, np.int32)
    cl = np.ascontiguousarray(cell_l, np.int32)
    n = cm.size
    out = np.empty(n, np.float64)
    rc = _load().kvo_eval_cells(_p(a["samples"]), _p(a["offsets"]), _p(a["L"]), _p(a["L_in"]), _p(a["r"]),
                                _p(a["lam"]), _p(a["cp"]), _p(a["cw"]), n, _p(cm), _p(ck), _p(cr), _p(cl),
                                _p(out), int(threads or default_threads()))
    if rc != 0:
        raise RuntimeError(f"kvo_eval_cells failed ({rc})")
    return out


def eval_grid(w, threads: Optional[int] = None) -> np.ndarray:
    """S[m, k, r, l] over the whole grid by the direct sample mean."""
    M, K, R, NL = len(w.cp), w.K, len(w.r), len(w.lam)
    mm, kk, rr, ll = np.meshgrid(np.arange(M), np.arange(K), np.arange(R), np.arange(NL), indexing="ij")
    S = eval_cells(w, mm.ravel(), kk.ravel(), rr.ravel(), ll.ravel(), threads)
    return S.reshape(M, K, R, NL)


def cumulative(w, k: int):
    """C[v] = #{x <= v}, Sx[v] = sum of x <= v for v = 0..L_k (exact int64)."""
    x = np.ascontiguousarray(w.class_samples(k), np.int32)
    L = int(w.L[k])
    C = np.empty(L + 1, np.int64)
    Sx = np.empty(L + 1, np.int64)
    if _load().kvo_cumulative(_p(x), x.size, L, _p(C), _p(Sx)) != 0:
        raise ValueError("sample outside [0, L]")
    return C, Sx


def envelope_grid(w, threads: Optional[int] = None) -> np.ndarray:
    """S[m, k, r, l] over the whole grid by the envelope regrouping (same sum, O(1) per cell)."""
    a = _arrays(w)
    K = w.K
    stride = int(w.L.max()) + 1
    C = np.zeros((K, stride), np.int64)
    Sx = np.zeros((K, stride), np.int64)
    for k in range(K):
        c, s = cumulative(w, k)
        C[k, :c.size] = c
        Sx[k, :s.size] = s
    N = np.ascontiguousarray(np.diff(w.offsets), np.int64)
    M, R, NL = len(w.cp), len(w.r), len(w.lam)
    out = np.empty((M, K, R, NL), np.float64)
    rc = _load().kvo_envelope_grid(_p(C), _p(Sx), stride, _p(N), _p(a["L"]), _p(a["L_in"]), _p(a["r"]),
                                   _p(a["lam"]), _p(a["cp"]), _p(a["cw"]), M, K, R, NL, _p(out),
                                   int(threads or default_threads()))
    if rc != 0:
        raise RuntimeError("kvo_envelope_grid failed")
    return out


def exact_dual_grid(w, threads: Optional[int] = None):
    """cost[m, e, k, r] = min over gamma >= 0 of gamma eps_e + S(eta, gamma) (App. A,
    eq. app_kantorovich without a grid) and a minimising gamma, by evaluating the convex
    piecewise-linear objective at gamma = 0 and at every kink of every sample's supremum."""
    a = _arrays(w)
    K = w.K
    stride = int(w.L.max()) + 1
    C = np.zeros((K, stride), np.int64)
    Sx = np.zeros((K, stride), np.int64)
    vals, voff = [], [0]
    for k in range(K):
        c, s_ = cumulative(w, k)
        C[k, :c.size] = c
        Sx[k, :s_.size] = s_
        u = np.unique(w.class_samples(k)).astype(np.int32)
        vals.append(u)
        voff.append(voff[-1] + u.size)
    vals = np.ascontiguousarray(np.concatenate(vals), np.int32)
    voff = np.ascontiguousarray(voff, np.int64)
    N = np.ascontiguousarray(np.diff(w.offsets), np.int64)
    eps = np.ascontiguousarray(w.eps, np.float64)
    M, E, R = len(w.cp), len(w.eps), len(w.r)
    cost = np.empty((M, E, K, R), np.float64)
    gam = np.empty((M, E, K, R), np.float64)
    rc = _load().kvo_exact_dual_grid(_p(C), _p(Sx), stride, _p(N), _p(a["L"]), _p(a["L_in"]), _p(vals), _p(voff),
                                     _p(a["r"]), _p(eps), _p(a["cp"]), _p(a["cw"]), M, E, K, R, _p(cost), _p(gam),
                                     int(threads or default_threads()))
    if rc != 0:
        raise RuntimeError("kvo_exact_dual_grid failed")
    return cost, gam


def solve_dual(w, threads: Optional[int] = None) -> Dict[str, np.ndarray]:
    """The exact dual cost, a minimising gamma, the argmin over r, its minimum and Fhat(r*)."""
    cost, gam = exact_dual_grid(w, threads)
    r_idx, min_cost = argmin_r(cost)
    return dict(cost=cost, gamma=gam, r_idx=r_idx, min_cost=min_cost, fhat=fhat_at(w, r_idx))


# ---------------------------------------------------------------- epilogue

def eps_epilogue(S: np.ndarray, lam: np.ndarray, eps: np.ndarray):
    """cost[m, e, k, r] = min_j (lam_j eps_e + S[m, k, r, j]) -- the dual objective of
    App. A (strong duality, gamma restricted to the lam grid); lam_idx is the lowest j
    attaining the minimum (reading: ties go to the lowest index).  One radius at a time."""
    lam = np.asarray(lam, np.float64)
    eps = np.asarray(eps, np.float64)
    M, K, R, NL = S.shape
    cost = np.empty((M, eps.size, K, R), np.float64)
    lam_idx = np.empty((M, eps.size, K, R), np.int32)
    for e, ep in enumerate(eps):
        obj = lam[None, None, None, :] * ep + S                 # [m, k, r, j]
        j = np.argmin(obj, axis=-1)                            # first occurrence = lowest index
        lam_idx[:, e] = j
        cost[:, e] = np.take_along_axis(obj, j[..., None], axis=-1)[..., 0]
    return cost, lam_idx


def argmin_r(cost: np.ndarray):
    """r_idx[m, e, k] = lowest r index attaining min_r cost[m, e, k, r]; also the minimum."""
    r_idx = np.argmin(cost, axis=-1).astype(np.int32)          # first occurrence = lowest index
    min_cost = np.take_along_axis(cost, r_idx[..., None].astype(np.int64), axis=-1)[..., 0]
    return r_idx, min_cost


def fhat_at(w, r_idx: np.ndarray) -> np.ndarray:
    """Empirical CDF at the chosen reservation, #{x <= r* - L_in} / N, per [m, e, k]
    (the "DRO quantile" that Fig. 3b plots against q*)."""
    out = np.empty(r_idx.shape, np.float64)
    for k in range(w.K):
        x = np.sort(w.class_samples(k))
        eta = w.r[r_idx[:, :, k]].astype(np.int64) - int(w.L_in[k])
        out[:, :, k] = np.searchsorted(x, eta, side="right") / x.size
    return out


def quantile_rank(q: float, n: int) -> int:
    """1-based order-statistic rank of the lower empirical q-quantile,
    max(1, ceil(q n)) computed in FP64 (reading: F^-1(q) = inf{x : F(x) >= q};
    q = 0 gives the minimum)."""
    return max(1, int(math.ceil(float(q) * float(n))))


def quantiles(w, fractiles: Sequence[float]) -> np.ndarray:
    """quant[k, f] = x_(m) with m = quantile_rank(q_f, N_k), from the sorted class
    samples (Prop. "Critical Fractile Structure", eq. critical_fractile)."""
    fr = np.asarray(fractiles, np.float64)
    out = np.empty((w.K, fr.size), np.int32)
    for k in range(w.K):
        xs = np.sort(w.class_samples(k), kind="stable")
        for f, q in enumerate(fr):
            out[k, f] = xs[quantile_rank(q, xs.size) - 1]
    return out


def solve(w, threads: Optional[int] = None, method: str = "direct") -> Dict[str, np.ndarray]:
    """Every output of one grid pass: S, cost, lam_idx, r_idx, min_cost, Fhat(r*), quantiles."""
    S = eval_grid(w, threads) if method == "direct" else envelope_grid(w, threads)
    cost, lam_idx = eps_epilogue(S, w.lam, w.eps)
    r_idx, min_cost = argmin_r(cost)
    return dict(S=S, cost=cost, lam_idx=lam_idx, r_idx=r_idx, min_cost=min_cost,
                fhat=fhat_at(w, r_idx), quant=quantiles(w, w.fractiles))
