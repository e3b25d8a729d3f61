"""CUDA path versus the oracle on the full-size synthetic workloads.

The envelope evaluator of the oracle (the same finite sum regrouped by affine pieces over
exact cumulative counts, pinned in test_oracle_pins.py) gives every cell of the full grids;
the direct per-term evaluator checks randomly drawn cells of the same runs.  The regime
sweep (all 1024 regimes) runs exactly as bench.py times it (FP32, the same outputs); the
8-class workload runs in FP32, exact and native FP64 over its full grid.
"""

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

from oracle import oracle as O
from synth import (drift_loop_workload_k32_n1e6, heavy_tail_workload_k16_n1e6, lognormal_workload_k8_n1e5,
                   regime_sweep_workload_k8_n2e5, slice_workload)
from tests.parity import RTOL, compare_full, oracle_from_S, rel_close

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402
from paper_2607_16892_gb300.runner import run  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def direct_cells(w, gpu_S, n, rtol, seed):
    """The direct per-term oracle on n random cells (plus each class's first and last r)."""
    rng = np.random.default_rng(seed)
    M, K, R, NL = gpu_S.shape
    m = rng.integers(0, M, n)
    k = rng.integers(0, K, n)
    r = rng.integers(0, R, n)
    l = rng.integers(0, NL, n)
    m = np.concatenate([m, np.zeros(2 * K, np.int64)])
    k = np.concatenate([k, np.repeat(np.arange(K), 2)])
    r = np.concatenate([r, np.tile([0, R - 1], K)])
    l = np.concatenate([l, rng.integers(0, NL, 2 * K)])
    ref = O.eval_cells(w, m, k, r, l)
    return rel_close(gpu_S[m, k, r, l], ref, rtol, "S (direct cells)")


def chosen_r_cells(w, gpu_S, gpu_r_idx, rtol, seed, max_terms=4e9):
    """The direct per-term oracle at every cell of each (regime, class)'s chosen reservations and
    their neighbours: r* and r* +- 1 over every radius, every lam value -- or, when that would pass
    max_terms terms, a seeded subset of the lam values that keeps each row's chosen ones."""
    rng = np.random.default_rng(seed)
    M, K, R, NL = gpu_S.shape
    cells = []
    for mm in range(M):
        for k in range(K):
            rs = np.unique(np.clip(np.concatenate([gpu_r_idx[mm, :, k] + d for d in (-1, 0, 1)]), 0, R - 1))
            for ri in rs:
                cells.append((mm, k, ri))
    cells = np.array(cells, np.int64)
    n_per = int(np.mean(w.N))
    keep = NL if len(cells) * NL * n_per <= max_terms else max(4, int(max_terms // (len(cells) * n_per)))
    m, k, r, l = [], [], [], []
    for mm, kk, ri in cells:
        lams = np.arange(NL) if keep >= NL else rng.choice(NL, keep, replace=False)
        m.append(np.full(len(lams), mm))
        k.append(np.full(len(lams), kk))
        r.append(np.full(len(lams), ri))
        l.append(lams)
    m, k, r, l = (np.concatenate(v) for v in (m, k, r, l))
    ref = O.eval_cells(w, m, k, r, l)
    return rel_close(gpu_S[m, k, r, l], ref, rtol, "S (cells at the chosen r)")


def test_lognormal_k8_n1e5_fp32_full_grid_as_benchmarked():
    w = lognormal_workload_k8_n1e5()
    gpu = run(w, kvdro.KVDRO_FP32)
    S_env = O.envelope_grid(w)
    rep = compare_full(w, gpu, oracle_from_S(w, S_env), "fp32")
    rep["direct"] = direct_cells(w, gpu["S"], 4096, RTOL["fp32"], 1)
    rep["direct_at_r_star"] = chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["fp32"], 11)
    assert rep["r_idx_exact"] > 0
    print(rep)


def test_lognormal_k8_n1e5_exact_full_grid():
    """The exact mode on every cell of the benchmarked grid, at the FP64 tolerance."""
    w = lognormal_workload_k8_n1e5()
    gpu = run(w, kvdro.KVDRO_EXACT)
    rep = compare_full(w, gpu, oracle_from_S(w, O.envelope_grid(w)), "exact")
    rep["direct"] = direct_cells(w, gpu["S"], 4096, RTOL["exact"], 7)
    rep["direct_at_r_star"] = chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["exact"], 17)
    print(rep)


def test_heavy_tail_k16_n1e6_exact_full_grid():
    w = heavy_tail_workload_k16_n1e6()
    gpu = run(w, kvdro.KVDRO_EXACT)
    rep = compare_full(w, gpu, oracle_from_S(w, O.envelope_grid(w)), "exact")
    rep["direct"] = direct_cells(w, gpu["S"], 4096, RTOL["exact"], 8)
    rep["direct_at_r_star"] = chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["exact"], 18)
    print(rep)


def test_lognormal_k8_n1e5_fp64_full_grid():
    """Native FP64 arithmetic per term on every cell of the 8-class grid (4096 r x 128 lam)."""
    w = lognormal_workload_k8_n1e5()
    gpu = run(w, kvdro.KVDRO_FP64)
    rep = compare_full(w, gpu, oracle_from_S(w, O.envelope_grid(w)), "fp64")
    rep["direct"] = direct_cells(w, gpu["S"], 4096, RTOL["fp64"], 2)
    rep["direct_at_r_star"] = chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["fp64"], 12)
    print(rep)


def test_heavy_tail_k16_n1e6_fp32_full_grid():
    w = heavy_tail_workload_k16_n1e6()
    gpu = run(w, kvdro.KVDRO_FP32)
    rep = compare_full(w, gpu, oracle_from_S(w, O.envelope_grid(w)), "fp32")
    rep["direct"] = direct_cells(w, gpu["S"], 4096, RTOL["fp32"], 3)
    rep["direct_at_r_star"] = chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["fp32"], 13)
    print(rep)


def test_regime_sweep_slice_and_critical_fractile():
    full = regime_sweep_workload_k8_n2e5()
    mi = np.arange(0, 1024, 16)  # 64 strided regimes, rho from 1 to ~900
    w = slice_workload(full, regimes=mi, name="regimes_slice")
    w.fractiles = (w.cp / (w.cp + w.cw)).copy()
    gpu = run(w, kvdro.KVDRO_FP32)
    ora = oracle_from_S(w, O.envelope_grid(w))
    compare_full(w, gpu, ora, "fp32")
    direct_cells(w, gpu["S"], 4096, RTOL["fp32"], 4)
    chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["fp32"], 14)
    _critical_fractile_rows(w, gpu["r_idx"], ora["cost"], ora["r_idx"], RTOL["fp32"])


def _critical_fractile_rows(w, gpu_r_idx, ora_cost, ora_r_idx, rtol):
    """eps = 0 (index 0): the oracle's argmin is the grid point at or next to each regime's
    critical-fractile quantile q = c_p / (c_p + c_w) (Prop. "Critical Fractile Structure"); the
    GPU's choice is that point too, or one whose oracle cost ties with it within rtol."""
    q = O.quantiles(w, w.cp / (w.cp + w.cw))  # [k, m]
    for mm in range(len(w.cp)):
        for k in range(w.K):
            lo = w.r[np.searchsorted(w.r, q[k, mm], side="right") - 1] if q[k, mm] >= w.r[0] else w.r[0]
            hi = w.r[min(np.searchsorted(w.r, q[k, mm], side="left"), len(w.r) - 1)]
            r_ora = w.r[ora_r_idx[mm, 0, k]]
            assert lo <= r_ora <= hi, (mm, k, r_ora, q[k, mm])
            g = gpu_r_idx[mm, 0, k]
            if not lo <= w.r[g] <= hi:
                row = ora_cost[mm, 0, k]
                assert row[g] <= row.min() * (1 + rtol), (mm, k, w.r[g], q[k, mm])


def test_regime_sweep_all_1024_regimes_as_benchmarked():
    """Every (regime, radius, class, r) of the regime sweep (8 classes x 200,000 samples, 2048 r,
    64 lam, 16 eps, 1024 cost ratios), run exactly as bench.py times it: cost, lam index, r index,
    minimum cost and F-hat against the oracle's envelope sums and eps epilogue, computed 16 regimes
    at a time on all host cores; the critical fractile at eps = 0 on every regime; quantiles."""
    w = regime_sweep_workload_k8_n2e5()
    gpu = run(w, kvdro.KVDRO_FP32, outputs=("cost", "lam_idx", "r_idx", "min_cost", "fhat", "quant"))
    assert np.array_equal(gpu["quant"], O.quantiles(w, w.fractiles))
    rtol = RTOL["fp32"]
    M = len(w.cp)
    step = 16

    def chunk(m0):
        mi = np.arange(m0, min(M, m0 + step))
        wc = slice_workload(w, regimes=mi, name=f"regimes_{m0}")
        ora = oracle_from_S(wc, O.envelope_grid(wc, threads=1))
        sub = {key: gpu[key][mi] for key in ("cost", "lam_idx", "r_idx", "min_cost", "fhat")}
        rep = compare_full(wc, sub, ora, "fp32")
        _critical_fractile_rows(wc, sub["r_idx"], ora["cost"], ora["r_idx"], rtol)
        return rep

    with ThreadPoolExecutor(max(1, min(16, os.cpu_count() or 1))) as ex:
        reps = list(ex.map(chunk, range(0, M, step)))
    print({"cost_max_rel": max(r["cost_max_rel"] for r in reps), "r_idx_exact": sum(r["r_idx_exact"] for r in reps),
           "lam_idx_exact": sum(r["lam_idx_exact"] for r in reps)})


@pytest.mark.parametrize("iteration", [0, 25, 49])
def test_drift_loop_k32_n1e6_iteration(iteration):
    w = drift_loop_workload_k32_n1e6(iteration)
    gpu = run(w, kvdro.KVDRO_FP32)
    rep = compare_full(w, gpu, oracle_from_S(w, O.envelope_grid(w)), "fp32")
    rep["direct"] = direct_cells(w, gpu["S"], 4096, RTOL["fp32"], 5 + iteration)
    rep["direct_at_r_star"] = chosen_r_cells(w, gpu["S"], gpu["r_idx"], RTOL["fp32"], 15 + iteration)
    print(rep)
