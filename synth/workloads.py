"""Seeded synthetic workloads.

The paper measures on production output-length traces (BurstGPT, Azure LLM
2024, ShareGPT; Sec. 5.1 "Trace Datasets").  Those traces are not available
here, so seeded lognormal and lognormal/Pareto mixtures with the shapes and
sizes of the five benchmark workloads stand in for them.  Every draw uses
``numpy.random.Generator(PCG64(seed))`` with

    seed = 20260000 + 1000 * workload_number + class_index (+ 100000 * iteration)

Samples are integers ``clip(rint(draw), 1, L)`` (output lengths in tokens),
stored per class in CSR form: ``offsets[K+1]`` (int64) and ``samples[offsets[K]]``
(int32).

Grid conventions (the paper does not fix them; they are the readings listed in
the design notes):
  * reservations ``r`` are integers on a uniform grid inside [L_in, L_in + L];
  * the dual-multiplier grid ``lam`` is log-spaced;
  * radii ``eps`` are in tokens (1-Wasserstein distance on token counts);
  * a cost regime is one (c_p, c_w) pair with c_w = 1 and c_p = rho.
"""

from __future__ import annotations

import dataclasses
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

SEED_BASE = 20260000


@dataclasses.dataclass
class Workload:
    """One evaluation problem: per-class samples plus the (r, lam, eps, regime) grid."""

    name: str
    samples: np.ndarray      # int32 [sum N_k], classes concatenated
    offsets: np.ndarray      # int64 [K+1], offsets[0] = 0
    L: np.ndarray            # int32 [K], support upper end per class
    L_in: np.ndarray         # int32 [K], input length per class
    r: np.ndarray            # int32 [R]
    lam: np.ndarray          # float64 [Lambda]
    eps: np.ndarray          # float64 [E]
    cp: np.ndarray           # float64 [M]
    cw: np.ndarray           # float64 [M]
    fractiles: np.ndarray    # float64 [F]
    precision: str = "fp32"  # arithmetic the workload is quoted in
    note: str = ""

    @property
    def K(self) -> int:
        return int(self.offsets.shape[0] - 1)

    @property
    def N(self) -> np.ndarray:
        return np.diff(self.offsets)

    def class_samples(self, k: int) -> np.ndarray:
        return self.samples[self.offsets[k]:self.offsets[k + 1]]

    def terms(self) -> int:
        """Cost terms of one grid pass: sum over classes of M * R * Lambda * N_k."""
        return int(len(self.cp) * len(self.r) * len(self.lam) * int(self.N.sum()))

    def sample_bytes(self) -> int:
        return int(self.samples.nbytes)


def _rng(workload_number: int, k: int, iteration: int = 0) -> np.random.Generator:
    seed = SEED_BASE + 1000 * workload_number + k + 100000 * iteration
    return np.random.Generator(np.random.PCG64(seed))


def _lognormal(rng: np.random.Generator, median: float, sigma: float, n: int, L: int) -> np.ndarray:
    z = rng.standard_normal(n)
    x = np.rint(np.exp(np.log(median) + sigma * z))
    return np.clip(x, 1, L).astype(np.int32)


def _lognormal_pareto_mix(rng: np.random.Generator, n: int, L: int, median: float = 200.0,
                          sigma: float = 0.7, x_min: float = 500.0, alpha: float = 1.3,
                          p_pareto: float = 0.3) -> np.ndarray:
    z = rng.standard_normal(n)
    u = rng.random(n)
    pick = rng.random(n) < p_pareto
    ln = np.exp(np.log(median) + sigma * z)
    # Pareto(x_min, alpha) by inversion; 1 - u lies in (0, 1].
    par = x_min * np.power(1.0 - u, -1.0 / alpha)
    x = np.rint(np.where(pick, par, ln))
    return np.clip(x, 1, L).astype(np.int32)


def _csr(classes: Sequence[np.ndarray]) -> (np.ndarray, np.ndarray):
    offsets = np.zeros(len(classes) + 1, dtype=np.int64)
    offsets[1:] = np.cumsum([len(c) for c in classes])
    samples = np.concatenate(classes).astype(np.int32) if classes else np.zeros(0, np.int32)
    return samples, offsets


def _logspace(lo: float, hi: float, n: int) -> np.ndarray:
    return np.logspace(np.log10(lo), np.log10(hi), n)


def lognormal_workload_k3_n1e3() -> Workload:
    """3 classes x 1,000 lognormal samples (medians 60/300/2000, sigma 0.8/0.9/1.0,
    clip [1, 8192]); r = 1 + 16 j (512 points); 32 lam in [1e-3, 1e2];
    eps in {0, 10, 100}; c_w = 1, c_p = 20; quoted in FP64."""
    L = 8192
    med, sig = [60.0, 300.0, 2000.0], [0.8, 0.9, 1.0]
    cls = [_lognormal(_rng(1, k), med[k], sig[k], 1000, L) for k in range(3)]
    samples, offsets = _csr(cls)
    return Workload(
        name="lognormal_k3_n1e3_r512_lam32_eps3",
        samples=samples, offsets=offsets,
        L=np.full(3, L, np.int32), L_in=np.zeros(3, np.int32),
        r=(1 + 16 * np.arange(512)).astype(np.int32),
        lam=_logspace(1e-3, 1e2, 32), eps=np.array([0.0, 10.0, 100.0]),
        cp=np.array([20.0]), cw=np.array([1.0]),
        fractiles=np.array([20.0 / 21.0, 0.5, 0.9, 0.95, 0.99]),
        precision="fp64")


def _k8_lognormal(workload_number: int, n: int, L: int = 32768, K: int = 8,
                  iteration: int = 0, drift: float = 1.0) -> List[np.ndarray]:
    med = _logspace(40.0, 4000.0, K) * drift
    sig = np.linspace(0.6, 1.2, K)
    return [_lognormal(_rng(workload_number, k, iteration), med[k], sig[k], n, L) for k in range(K)]


def lognormal_workload_k8_n1e5() -> Workload:
    """8 classes x 100,000 lognormal samples (medians log-spaced 40..4000, sigma
    linear 0.6..1.2, clip [1, 32768]); r = 8 (j+1) (4096 points); 128 lam in
    [1e-3, 1e2]; 8 eps log-spaced 1..1000; c_w = 1, c_p = 10."""
    L = 32768
    samples, offsets = _csr(_k8_lognormal(2, 100_000, L))
    return Workload(
        name="lognormal_k8_n1e5_r4096_lam128_eps8",
        samples=samples, offsets=offsets,
        L=np.full(8, L, np.int32), L_in=np.zeros(8, np.int32),
        r=(8 * (np.arange(4096) + 1)).astype(np.int32),
        lam=_logspace(1e-3, 1e2, 128), eps=_logspace(1.0, 1000.0, 8),
        cp=np.array([10.0]), cw=np.array([1.0]),
        fractiles=np.array([10.0 / 11.0, 0.5, 0.9, 0.95, 0.99]),
        precision="fp32")


def heavy_tail_workload_k16_n1e6() -> Workload:
    """16 classes x 1,000,000 samples of a 70/30 mixture of lognormal(median 200,
    sigma 0.7) and Pareto(x_min 500, alpha 1.3), clip [1, 131072]; r = 16 (j+1)
    (8192 points); 128 lam in [1e-3, 1e2]; eps in {0, 50, 500}; c_w = 1, c_p = 10."""
    L = 131072
    cls = [_lognormal_pareto_mix(_rng(3, k), 1_000_000, L) for k in range(16)]
    samples, offsets = _csr(cls)
    return Workload(
        name="heavytail_k16_n1e6_r8192_lam128_eps3",
        samples=samples, offsets=offsets,
        L=np.full(16, L, np.int32), L_in=np.zeros(16, np.int32),
        r=(16 * (np.arange(8192) + 1)).astype(np.int32),
        lam=_logspace(1e-3, 1e2, 128), eps=np.array([0.0, 50.0, 500.0]),
        cp=np.array([10.0]), cw=np.array([1.0]),
        fractiles=np.array([10.0 / 11.0, 0.5, 0.9, 0.95, 0.99]),
        precision="fp32")


def regime_sweep_workload_k8_n2e5() -> Workload:
    """8 classes x 200,000 lognormal samples as in the k8 workload; 1024 regimes
    with c_w = 1 and c_p = rho log-spaced over [1, 1000]; eps = {0} plus 15
    log-spaced in [1, 1000]; r = 16 (j+1) (2048 points); 64 lam in [1e-3, 1e3]."""
    L = 32768
    samples, offsets = _csr(_k8_lognormal(4, 200_000, L))
    rho = _logspace(1.0, 1000.0, 1024)
    return Workload(
        name="regimes_k8_n2e5_m1024_r2048_lam64_eps16",
        samples=samples, offsets=offsets,
        L=np.full(8, L, np.int32), L_in=np.zeros(8, np.int32),
        r=(16 * (np.arange(2048) + 1)).astype(np.int32),
        lam=_logspace(1e-3, 1e3, 64),
        eps=np.concatenate([[0.0], _logspace(1.0, 1000.0, 15)]),
        cp=rho.copy(), cw=np.ones(1024),
        fractiles=rho / (rho + 1.0),
        precision="fp32")


def drift_loop_workload_k32_n1e6(iteration: int = 0) -> Workload:
    """One iteration of the drifting-median loop: 32 classes x 1,000,000 lognormal
    samples with medians log-spaced 40..4000 times 1.02**iteration, sigma linear
    0.6..1.2, clip [1, 32768], redrawn per iteration; r = 8 (j+1) (4096 points);
    128 lam in [1e-3, 1e2]; 8 eps log-spaced 1..1000; 64 fractiles; c_p = 10."""
    L = 32768
    cls = _k8_lognormal(5, 1_000_000, L, K=32, iteration=iteration, drift=1.02 ** iteration)
    samples, offsets = _csr(cls)
    return Workload(
        name=f"drift_k32_n1e6_r4096_lam128_eps8_it{iteration}",
        samples=samples, offsets=offsets,
        L=np.full(32, L, np.int32), L_in=np.zeros(32, np.int32),
        r=(8 * (np.arange(4096) + 1)).astype(np.int32),
        lam=_logspace(1e-3, 1e2, 128), eps=_logspace(1.0, 1000.0, 8),
        cp=np.array([10.0]), cw=np.array([1.0]),
        fractiles=np.linspace(0.0, 1.0, 64),
        precision="fp32")


WORKLOADS: Dict[str, Callable[[], Workload]] = {
    "lognormal_k3_n1e3": lognormal_workload_k3_n1e3,
    "lognormal_k8_n1e5": lognormal_workload_k8_n1e5,
    "heavytail_k16_n1e6": heavy_tail_workload_k16_n1e6,
    "regimes_k8_n2e5": regime_sweep_workload_k8_n2e5,
    "drift_k32_n1e6": drift_loop_workload_k32_n1e6,
}


def slice_workload(w: Workload, classes: Optional[Sequence[int]] = None,
                   r_index: Optional[Sequence[int]] = None,
                   regimes: Optional[Sequence[int]] = None,
                   n_per_class: Optional[int] = None, name: Optional[str] = None) -> Workload:
    """A sub-problem of ``w``: a subset of classes, r points, regimes, and/or the
    first ``n_per_class`` samples of every kept class (for bounded oracle runs)."""
    ks = list(range(w.K)) if classes is None else list(classes)
    cls = [w.class_samples(k) for k in ks]
    if n_per_class is not None:
        cls = [c[:n_per_class] for c in cls]
    samples, offsets = _csr(cls)
    ri = np.arange(len(w.r)) if r_index is None else np.asarray(r_index)
    mi = np.arange(len(w.cp)) if regimes is None else np.asarray(regimes)
    return Workload(
        name=name or (w.name + "_slice"),
        samples=samples, offsets=offsets,
        L=w.L[ks].copy(), L_in=w.L_in[ks].copy(),
        r=w.r[ri].copy(), lam=w.lam.copy(), eps=w.eps.copy(),
        cp=w.cp[mi].copy(), cw=w.cw[mi].copy(),
        fractiles=w.fractiles.copy(), precision=w.precision, note=w.note)


def random_case(seed: int, K: int = 3, N: Sequence[int] = (200, 77, 31), L: Sequence[int] = (600, 600, 600),
                L_in: Optional[Sequence[int]] = None, R: int = 37, n_lam: int = 21, n_eps: int = 3,
                M: int = 2, lam_range=(1e-2, 50.0), eps_max: float = 200.0, integer_costs: bool = False,
                r_grid: str = "uniform", fractiles: Optional[Sequence[float]] = None) -> Workload:
    """A small seeded case with ragged sizes: lognormal classes with random medians,
    an r grid inside every class's domain, random regimes, a log-spaced lam grid."""
    rng = np.random.Generator(np.random.PCG64(SEED_BASE + 900000 + seed))
    N = list(N)[:K]
    L = np.asarray(list(L)[:K], np.int32)
    Lin = np.zeros(K, np.int32) if L_in is None else np.asarray(list(L_in)[:K], np.int32)
    cls = []
    for k in range(K):
        med = float(np.exp(rng.uniform(np.log(5.0), np.log(max(6.0, 0.4 * L[k])))))
        sig = float(rng.uniform(0.4, 1.3))
        z = rng.standard_normal(N[k])
        cls.append(np.clip(np.rint(np.exp(np.log(med) + sig * z)), 1, L[k]).astype(np.int32))
    samples, offsets = _csr(cls)
    lo = int(Lin.max())
    hi = int((Lin + L).min())
    if r_grid == "uniform":
        r = np.unique(np.linspace(lo, hi, R).round().astype(np.int64)).astype(np.int32)
    else:
        r = np.sort(rng.integers(lo, hi + 1, R)).astype(np.int32)
    if integer_costs:
        cp = rng.integers(1, 30, M).astype(np.float64)
        cw = rng.integers(1, 4, M).astype(np.float64)
    else:
        cp = np.exp(rng.uniform(np.log(0.5), np.log(100.0), M))
        cw = np.exp(rng.uniform(np.log(0.2), np.log(3.0), M))
    lam = np.logspace(np.log10(lam_range[0]), np.log10(lam_range[1]), n_lam)
    eps = np.concatenate([[0.0], np.sort(rng.uniform(0.0, eps_max, max(0, n_eps - 1)))])
    fr = np.array([0.0, 0.1, 0.5, 0.9, 0.99, 1.0]) if fractiles is None else np.asarray(fractiles, np.float64)
    return Workload(name=f"random_case_{seed}", samples=samples, offsets=offsets, L=L, L_in=Lin,
                    r=r, lam=lam, eps=eps, cp=cp, cw=cw, fractiles=fr, precision="fp64")
