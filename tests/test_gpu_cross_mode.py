"""The library's modes against each other (no oracle): the per-term exact kernel and the O(1)-per-cell
envelope reach the same S by different algorithms; the exact dual, a minimum over every gamma >= 0,
can only be below the minimum over a lam grid, and meets it at eps = 0 once the grid reaches
max(c_p, c_w) (the saturated multiplier, App. A)."""

import numpy as np
import pytest

from synth import random_case

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402
from paper_2607_16892_gb300.runner import run  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def dual_cost(w):
    M, E, K, R = len(w.cp), len(w.eps), w.K, len(w.r)
    ctx = kvdro.kvdro_create(0)
    try:
        kvdro.kvdro_load_samples(ctx, K, w.offsets, torch.from_numpy(w.samples).cuda(), w.L, w.L_in)
        cost = np.empty((M, E, K, R), np.float64)
        kvdro.kvdro_eval_dual(ctx, R, w.r, E, w.eps, M, w.cp, w.cw, cost=cost)
    finally:
        kvdro.kvdro_destroy(ctx)
    return cost


@pytest.mark.parametrize("seed", range(8))
def test_exact_envelope_and_dual_agree(seed):
    rng = np.random.default_rng(seed)
    K = int(rng.integers(1, 5))
    N = tuple(int(v) for v in rng.integers(1, 6000, K))
    L = tuple(int(v) for v in rng.choice([50, 700, 4096, 20000], K))
    L_in = tuple(int(v) for v in rng.integers(0, min(L) // 2 + 1, K))  # keeps a common r domain
    # the lam grid reaches past every c_p and c_w (at most 100 and 3 here)
    w = random_case(1000 + seed, K=K, N=N, L=L, L_in=L_in, R=int(rng.integers(5, 60)), n_lam=int(rng.integers(8, 200)),
                    n_eps=4, M=int(rng.integers(1, 4)), lam_range=(1e-3, 200.0), eps_max=float(rng.uniform(10, 5000)),
                    integer_costs=bool(seed % 2))
    ex, env = run(w, kvdro.KVDRO_EXACT), run(w, kvdro.KVDRO_ENVELOPE)
    np.testing.assert_allclose(ex["S"], env["S"], rtol=1e-12, atol=0)
    np.testing.assert_allclose(ex["cost"], env["cost"], rtol=1e-12, atol=0)
    np.testing.assert_array_equal(ex["quant"], env["quant"])
    dual = dual_cost(w)
    grid = ex["cost"]
    assert np.all(dual <= grid * (1 + 1e-12) + 1e-12)                   # a minimum over more multipliers
    np.testing.assert_allclose(dual[:, 0], grid[:, 0], rtol=1e-11, atol=0)  # eps = 0: both are the empirical cost
