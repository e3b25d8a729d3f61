"""Exact dual (kvdro_eval_dual) and the envelope mode of kvdro_eval_grid against the oracle."""

import numpy as np
import pytest

from oracle import oracle as O
from synth import lognormal_workload_k3_n1e3, lognormal_workload_k8_n1e5, random_case, slice_workload
from tests.parity import RTOL, check_argmin, compare_full, oracle_from_S, rel_close

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402
from paper_2607_16892_gb300.runner import run  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def run_dual(w, host=False):
    dev = torch.device("cuda", 0)
    M, E, K, R = len(w.cp), len(w.eps), w.K, len(w.r)
    ctx = kvdro.kvdro_create(0)
    try:
        kvdro.kvdro_load_samples(ctx, K, w.offsets, torch.from_numpy(w.samples).to(dev), w.L, w.L_in)
        mk = (lambda shape, dt: np.empty(shape, dt)) if host else \
            (lambda shape, dt: torch.empty(shape, dtype=getattr(torch, np.dtype(dt).name), device=dev))
        out = dict(cost=mk((M, E, K, R), np.float64), gamma=mk((M, E, K, R), np.float64),
                   r_idx=mk((M, E, K), np.int32), min_cost=mk((M, E, K), np.float64), fhat=mk((M, E, K), np.float64))
        kvdro.kvdro_eval_dual(ctx, R, w.r, E, w.eps, M, w.cp, w.cw, **out)
        torch.cuda.synchronize()
        return {k: (v if isinstance(v, np.ndarray) else v.cpu().numpy()) for k, v in out.items()}
    finally:
        kvdro.kvdro_destroy(ctx)


def check_dual(w, gpu, ora, n_gamma=64, seed=0):
    rtol = RTOL["fp64"]
    rel_close(gpu["cost"], ora["cost"], rtol, "dual cost")
    rel_close(gpu["min_cost"], ora["min_cost"], rtol, "dual min cost")
    check_argmin(gpu["r_idx"], ora["cost"], rtol, "dual r_idx")
    for k in range(w.K):
        xs = np.sort(w.class_samples(k))
        eta = w.r[gpu["r_idx"][:, :, k]].astype(np.int64) - int(w.L_in[k])
        assert np.array_equal(gpu["fhat"][:, :, k], np.searchsorted(xs, eta, side="right") / xs.size)
    # the returned gamma attains the cost: g(gamma) by the direct per-sample oracle on sampled cells
    rng = np.random.default_rng(seed)
    M, E, K, R = gpu["cost"].shape
    for _ in range(n_gamma):
        m, e, k, i = (int(rng.integers(0, n)) for n in (M, E, K, R))
        gam = gpu["gamma"][m, e, k, i]
        assert 0.0 <= gam <= max(w.cp[m], w.cw[m])
        eta = float(w.r[i] - w.L_in[k])
        g = gam * w.eps[e] + O.mean_sup(w.class_samples(k), eta, gam, w.cp[m], w.cw[m], float(w.L[k]))
        assert abs(g - ora["cost"][m, e, k, i]) <= rtol * max(1.0, abs(ora["cost"][m, e, k, i]))


@pytest.mark.parametrize("seed", [41, 42])
def test_dual_random_ragged(seed):
    w = random_case(seed, K=3, N=(3000, 411, 17), L=(2500, 2500, 2500), R=31, n_lam=4, n_eps=5, M=3,
                    eps_max=3000.0)
    check_dual(w, run_dual(w), O.solve_dual(w), seed=seed)


def test_dual_per_class_support_host_outputs():
    w = random_case(43, K=3, N=(900, 77, 5), L=(700, 900, 1200), L_in=(0, 20, 5), R=17, n_lam=3, n_eps=3, M=2,
                    integer_costs=True)
    a, b = run_dual(w), run_dual(w, host=True)
    for k in a:
        assert np.array_equal(a[k], b[k]), k
    check_dual(w, a, O.solve_dual(w))


def test_dual_lognormal_k3_n1e3_and_below_the_grid():
    w = lognormal_workload_k3_n1e3()
    d = run_dual(w)
    check_dual(w, d, O.solve_dual(w))
    grid = run(w, kvdro.KVDRO_FP64, outputs=("cost",))
    assert np.all(d["cost"] <= grid["cost"] * (1 + 1e-12))


def test_dual_lognormal_k8_n1e5_slice():
    w = slice_workload(lognormal_workload_k8_n1e5(), r_index=np.arange(5, 4096, 128), name="k8_dual_slice")
    check_dual(w, run_dual(w), O.solve_dual(w), n_gamma=16)


@pytest.mark.parametrize("seed", [1, 2])
def test_envelope_mode_random_ragged(seed):
    w = random_case(seed, K=3, N=(5000, 777, 33), L=(3000, 3000, 3000), R=45, n_lam=37, n_eps=4, M=3,
                    lam_range=(1e-3, 200.0), eps_max=300.0)
    compare_full(w, run(w, kvdro.KVDRO_ENVELOPE), O.solve(w), "fp64")


def test_envelope_mode_edge_cases():
    rng = np.random.default_rng(3)
    w = random_case(9, K=4, N=(2100, 129, 128, 1), L=(900, 1500, 2000, 1200), L_in=(0, 50, 10, 200), R=33,
                    n_lam=256, n_eps=3, M=2, lam_range=(1e-4, 1e3))
    compare_full(w, run(w, kvdro.KVDRO_ENVELOPE), O.solve(w), "fp64")
    w.lam = np.concatenate([[0.0], w.lam[1:]])
    compare_full(w, run(w, kvdro.KVDRO_ENVELOPE), O.solve(w), "fp64")


def test_envelope_mode_lognormal_k8_n1e5_full_grid():
    w = lognormal_workload_k8_n1e5()
    gpu = run(w, kvdro.KVDRO_ENVELOPE)
    compare_full(w, gpu, oracle_from_S(w, O.envelope_grid(w)), "fp64")
    rng = np.random.default_rng(11)
    m = np.zeros(256, np.int64)
    k, r, l = rng.integers(0, w.K, 256), rng.integers(0, len(w.r), 256), rng.integers(0, len(w.lam), 256)
    rel_close(gpu["S"][m, k, r, l], O.eval_cells(w, m, k, r, l), RTOL["fp64"], "S (direct cells)")


def exact_empirical_cost(w):
    """(1/N) sum_n Q(eta, x_n) per [m, k, r], exact (integer sums, c_p and c_w as fractions) and
    rounded once: the dual's value at eps = 0 and a lower bound at every eps, since the empirical
    distribution lies in every Wasserstein ball (App. A)."""
    from fractions import Fraction
    M, K, R = len(w.cp), w.K, len(w.r)
    out = np.empty((M, K, R), np.float64)
    for k in range(K):
        x = [int(v) for v in w.class_samples(k)]
        for i in range(R):
            eta = int(w.r[i]) - int(w.L_in[k])
            below = sum(eta - v for v in x if v < eta)
            above = sum(v - eta for v in x if v > eta)
            for m in range(M):
                out[m, k, i] = float((Fraction(w.cw[m]) * below + Fraction(w.cp[m]) * above) / len(x))
    return out


def check_dual_scaled(w, gpu, ora):
    """The dual with c_p and c_w many orders apart.  Its minimiser sits where two of phi's lines
    cross, lines of size up to c_w eta + c_p (L - eta) + max(c_p, c_w) L; FP64 places a sample at such
    a crossing only to within eps times that size (the oracle's crossing points as the kernel's
    thresholds), so a cell compares within rtol plus 16 eps times that size.  The exact bounds hold
    whatever the scale: cost >= the empirical cost, with equality at eps = 0."""
    rtol = RTOL["fp64"]
    M, E, K, R = gpu["cost"].shape
    cp, cw = np.asarray(w.cp)[:, None, None, None], np.asarray(w.cw)[:, None, None, None]
    eta = (w.r[None, :].astype(np.float64) - w.L_in[:, None].astype(np.float64))[None, None]  # [1, 1, K, R]
    L = w.L.astype(np.float64)[None, None, :, None]
    size = cw * eta + cp * (L - eta) + np.maximum(cp, cw) * L
    tol = rtol * np.abs(ora["cost"]) + 16 * np.finfo(np.float64).eps * size
    err = np.abs(gpu["cost"] - ora["cost"])
    assert np.all(err <= tol), (np.argmax(err - tol), gpu["cost"].ravel()[np.argmax(err - tol)])
    emp = exact_empirical_cost(w)[:, None]                                       # [M, 1, K, R]
    assert np.all(gpu["cost"] >= emp * (1 - 4 * np.finfo(np.float64).eps)), "below the empirical cost"
    at0 = np.asarray(w.eps) == 0.0
    np.testing.assert_allclose(gpu["cost"][:, at0], np.broadcast_to(emp, gpu["cost"].shape)[:, at0], rtol=4e-15, atol=0)
    # the chosen reservation is a minimiser within the same tolerance
    chosen = np.take_along_axis(ora["cost"], gpu["r_idx"][..., None].astype(np.int64), axis=-1)[..., 0]
    assert np.all(chosen <= ora["cost"].min(axis=-1) + tol.max(axis=-1))
    np.testing.assert_array_equal(gpu["min_cost"], np.take_along_axis(gpu["cost"], gpu["r_idx"][..., None].astype(np.int64), axis=-1)[..., 0])


@pytest.mark.parametrize("scale", ["tiny", "huge"])
def test_dual_costs_far_outside_fp32_range(scale):
    """The exact dual with c_w or c_p many orders apart (tiny: down to 1e-300; huge: up to 1e150)."""
    rng = np.random.default_rng(23)
    from tests.test_gpu_parity import make
    if scale == "tiny":
        w = make([rng.integers(0, 300, 2000), rng.integers(100, 301, 60)], 300, [0, 7, 150, 299, 300], [1.0],
                 [0.0, 1e-10, 3.0], [10.0, 1e-300, 2.0], [1.0, 1e-300, 1e-250])
    else:
        w = make([rng.integers(0, 5000, 1500), rng.integers(4000, 5001, 40)], 5000, [0, 1, 2500, 4999, 5000], [1.0],
                 [0.0, 1.0, 1e100], [1e150, 1.0, 2e150], [1.0, 1e150, 5e149])
    check_dual_scaled(w, run_dual(w), O.solve_dual(w))


@pytest.mark.parametrize("seed", range(4))
def test_dual_equals_the_empirical_cost_at_eps_zero(seed):
    """At eps = 0 the worst case over the ball is the empirical cost itself (App. A), for any costs."""
    rng = np.random.default_rng(300 + seed)
    w = random_case(300 + seed, K=3, N=(int(rng.integers(1, 3000)), 57, 1), L=(1000, 4096, 300), R=17, n_lam=4,
                    n_eps=3, M=3, lam_range=(1e-3, 200.0), eps_max=50.0)
    w.eps[0] = 0.0
    gpu = run_dual(w)
    emp = exact_empirical_cost(w)
    np.testing.assert_allclose(gpu["cost"][:, 0], emp, rtol=4e-15, atol=0)  # a few roundings
    assert np.all(gpu["cost"] >= emp[:, None] * (1 - 4 * np.finfo(np.float64).eps))

