"""The seeded synthetic inputs follow the recipe the workloads are quoted with (sizes, supports,
grids, costs, and the distributions' own statistics): lognormal medians and spreads, the 70/30
lognormal-Pareto mixture of the heavy-tail workload, and the drift of the loop workload's medians.
The statistics are checked against their closed forms with margins of several standard errors."""

import math

import numpy as np
import pytest

from synth import WORKLOADS, drift_loop_workload_k32_n1e6


def _logspace(lo, hi, n):
    return np.logspace(math.log10(lo), math.log10(hi), n)


def _median_and_sigma(x):
    """Sample median and the lognormal sigma from the interquartile range of log x (the middle
    half of every class here lies inside its clip range)."""
    lx = np.log(x.astype(np.float64))
    q25, q50, q75 = np.percentile(lx, [25, 50, 75])
    return math.exp(q50), (q75 - q25) / 1.3489795003921634


def _check_grid(w, K, N, L, r, lam, eps, cp, cw):
    assert w.K == K and np.all(w.N == N)
    assert np.all(w.L == L) and np.all(w.L_in == 0)
    assert w.samples.dtype == np.int32 and w.samples.min() >= 1 and w.samples.max() <= L
    np.testing.assert_array_equal(w.r, r)
    np.testing.assert_allclose(w.lam, lam, rtol=1e-12)
    np.testing.assert_allclose(w.eps, eps, rtol=1e-12)
    np.testing.assert_allclose(w.cp, cp, rtol=1e-12)
    np.testing.assert_allclose(w.cw, cw, rtol=1e-12)


def test_lognormal_k3_n1e3():
    w = WORKLOADS["lognormal_k3_n1e3"]()
    _check_grid(w, 3, 1000, 8192, 1 + 16 * np.arange(512), _logspace(1e-3, 1e2, 32), [0.0, 10.0, 100.0], [20.0], [1.0])
    for k, (med, sig) in enumerate(zip((60.0, 300.0, 2000.0), (0.8, 0.9, 1.0))):
        m, s = _median_and_sigma(w.class_samples(k))
        assert abs(math.log(m / med)) < 4 * 1.2533 * sig / math.sqrt(1000), (k, m)
        assert abs(s / sig - 1) < 0.15, (k, s)


@pytest.mark.parametrize("name,n,r", [("lognormal_k8_n1e5", 100_000, 8 * (np.arange(4096) + 1)),
                                      ("regimes_k8_n2e5", 200_000, 16 * (np.arange(2048) + 1))])
def test_lognormal_k8_classes(name, n, r):
    w = WORKLOADS[name]()
    if name == "lognormal_k8_n1e5":
        _check_grid(w, 8, n, 32768, r, _logspace(1e-3, 1e2, 128), _logspace(1, 1000, 8), [10.0], [1.0])
    else:  # 1024 cost regimes c_p / c_w = rho log-spaced over [1, 1000]; eps 0 plus 15 log-spaced
        rho = _logspace(1, 1000, 1024)
        _check_grid(w, 8, n, 32768, r, _logspace(1e-3, 1e3, 64), np.concatenate([[0.0], _logspace(1, 1000, 15)]),
                    rho, np.ones(1024))
        np.testing.assert_allclose(w.fractiles, rho / (rho + 1), rtol=1e-12)
    meds, sigs = _logspace(40, 4000, 8), np.linspace(0.6, 1.2, 8)
    for k in range(8):
        m, s = _median_and_sigma(w.class_samples(k))
        # the median of rounded samples: within the standard error, plus half a token of rounding
        assert abs(m - meds[k]) < 4 * 1.2533 * sigs[k] * meds[k] / math.sqrt(n) + 0.5, (k, m)
        assert abs(s / sigs[k] - 1) < 0.03 + 0.5 / meds[k], (k, s)


def test_heavy_tail_mixture():
    w = WORKLOADS["heavytail_k16_n1e6"]()
    _check_grid(w, 16, 1_000_000, 131072, 16 * (np.arange(8192) + 1), _logspace(1e-3, 1e2, 128), [0.0, 50.0, 500.0],
                [10.0], [1.0])
    # P(x >= 500): the whole Pareto share plus the lognormal(200, 0.7) tail above 500
    ln_tail = 0.5 * math.erfc(math.log(500 / 200) / 0.7 / math.sqrt(2))
    p500 = 0.3 + 0.7 * ln_tail
    # P(x >= 5000): the Pareto(500, 1.3) share (the lognormal part is below 1e-5 there)
    p5000 = 0.3 * (500 / 5000) ** 1.3
    for k in range(16):
        x = w.class_samples(k)
        f500 = np.mean(x >= 500)   # rounding moves at most the samples within half a token of 500
        f5000 = np.mean(x >= 5000)
        assert abs(f500 - p500) < 5 * math.sqrt(p500 * (1 - p500) / x.size) + 2e-4, (k, f500, p500)
        assert abs(f5000 - p5000) < 5 * math.sqrt(p5000 * (1 - p5000) / x.size), (k, f5000, p5000)
        assert x.max() == 131072  # the Pareto tail reaches the clip


def test_drift_loop_medians_move_by_two_percent_per_iteration():
    w0 = drift_loop_workload_k32_n1e6(0)
    w10 = drift_loop_workload_k32_n1e6(10)
    r = 8 * (np.arange(4096) + 1)
    for w in (w0, w10):
        _check_grid(w, 32, 1_000_000, 32768, r, _logspace(1e-3, 1e2, 128), _logspace(1, 1000, 8), [10.0], [1.0])
        assert len(w.fractiles) == 64
    meds, sigs = _logspace(40, 4000, 32), np.linspace(0.6, 1.2, 32)
    for k in (0, 11, 31):
        for w, t in ((w0, 0), (w10, 10)):
            m, _ = _median_and_sigma(w.class_samples(k))
            want = meds[k] * 1.02 ** t
            assert abs(m - want) < 4 * 1.2533 * sigs[k] * want / 1000 + 0.5, (k, t, m, want)
    assert not np.array_equal(w0.class_samples(0), w10.class_samples(0))  # redrawn per iteration
