"""Worst-case cost tables for the block-coordinate-descent tests, computed by the oracle."""

from __future__ import annotations

import numpy as np

from oracle import oracle as O
from paper_2607_16892_gb300 import bcd
from synth import Workload


def oracle_tables(p: bcd.Problem) -> bcd.Tables:
    """f_i(eta) = min over gamma >= 0 of gamma eps_i + S_i(eta, gamma) for eta = 0..L_max^i (the
    oracle's exact dual by kink enumeration) and the initial point's cost at gamma = c_p
    (c_p eps_i + the oracle's envelope sum), laid out as ``bcd.gpu_tables`` lays them out."""
    I = p.I
    Lmax = int(p.L_max.max())
    cost = np.full((I, Lmax + 1), np.inf)
    gamma = np.full((I, Lmax + 1), np.nan)
    eta0 = np.clip(np.rint(p.mean_output()), 0, p.L_max).astype(np.int64)
    d0 = np.empty(I)
    for L in np.unique(p.L_max):
        idx = np.flatnonzero(p.L_max == L)
        n = idx.size
        parts = [p.class_samples(i) for i in idx]
        off = np.zeros(n + 1, np.int64)
        off[1:] = np.cumsum([x.size for x in parts])
        w = Workload(name="bcd", samples=np.concatenate(parts).astype(np.int32), offsets=off,
                     L=np.full(n, L, np.int32), L_in=np.zeros(n, np.int32), r=np.arange(L + 1, dtype=np.int32),
                     lam=np.array([p.c_p]), eps=np.asarray(p.eps[idx], np.float64), cp=np.array([p.c_p]),
                     cw=np.array([p.c_w]), fractiles=np.array([0.5]))
        c, g = O.exact_dual_grid(w)
        e0 = np.unique(eta0[idx]).astype(np.int32)
        w.r = e0
        S = O.envelope_grid(w)
        for j, i in enumerate(idx):
            cost[i, :L + 1] = c[0, j, j]
            gamma[i, :L + 1] = g[0, j, j]
            d0[i] = p.c_p * p.eps[i] + S[0, j, int(np.searchsorted(e0, eta0[i])), 0]
    return bcd.Tables(cost=cost, gamma=gamma, eta0=eta0, d0=d0)
