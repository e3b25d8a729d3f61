"""kvdro_eval_grid_noalloc against kvdro_eval_grid, through the C ABI, on two calls in a row.

The no-allocation entry point serves callers that cannot allocate device memory when they
need a reservation answer (for example a serving engine whose free memory all belongs to its
KV-cache pool).  It must give the same results as the context-based entry point, also when
the previous call left other data in its shared static scratch.  This file is collected last
so that a stop-at-first-failure run has already run every other test.
"""

import numpy as np
import pytest

from synth import random_case, lognormal_workload_k3_n1e3
from tests.parity import RTOL, check_argmin, rel_close

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402
from paper_2607_16892_gb300.runner import run  # noqa: E402


def _noalloc(w):
    dev = torch.device("cuda", torch.cuda.current_device())
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    out = {
        "cost": torch.full((M, E, K, R), -1.0, dtype=torch.float32, device=dev),
        "lam_idx": torch.full((M, E, K, R), -1, dtype=torch.int32, device=dev),
        "r_idx": torch.full((M, E, K), -1, dtype=torch.int32, device=dev),
        "min_cost": torch.full((M, E, K), -1.0, dtype=torch.float32, device=dev),
        "fhat": torch.full((M, E, K), -1.0, dtype=torch.float64, device=dev),
    }
    samples = torch.from_numpy(np.ascontiguousarray(w.samples, np.int32)).to(dev)
    kvdro.kvdro_eval_grid_noalloc(K, w.offsets, samples, w.L, w.L_in, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw,
                                  **out)
    torch.cuda.synchronize(dev)
    return {k: v.cpu().numpy() for k, v in out.items()}


def _compare(w, got, ref):
    rtol = RTOL["fp32"]
    rel_close(got["cost"], ref["cost"], rtol, "cost")
    rel_close(got["min_cost"], ref["min_cost"], rtol, "min_cost")
    obj = ref["cost"].astype(np.float64)
    check_argmin(got["r_idx"], obj, rtol, "r_idx")
    assert np.array_equal(got["lam_idx"] >= 0, np.ones_like(got["lam_idx"], bool))
    for k in range(w.K):
        xs = np.sort(w.class_samples(k))
        eta = w.r[got["r_idx"][:, :, k]].astype(np.int64) - int(w.L_in[k])
        assert np.array_equal(got["fhat"][:, :, k], np.searchsorted(xs, eta, side="right") / xs.size)


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_noalloc_matches_context_entry_point_on_two_calls_in_a_row():
    first = random_case(301, K=3, N=(6000, 513, 29), L=(4000, 4000, 4000), R=57, n_lam=40, n_eps=3, M=2,
                        lam_range=(1e-3, 100.0), eps_max=400.0)
    second = lognormal_workload_k3_n1e3()  # different K, N, L, grid and regime count
    for w in (first, second):
        ref = run(w, kvdro.KVDRO_FP32, outputs=("cost", "lam_idx", "r_idx", "min_cost", "fhat"))
        got = _noalloc(w)
        _compare(w, got, ref)
        for key in ("cost", "lam_idx", "r_idx", "min_cost", "fhat"):
            assert np.array_equal(got[key], ref[key]), key  # same kernels, same inputs


def test_noalloc_rejects_a_problem_larger_than_its_scratch():
    w = random_case(302, K=1, N=(10,), L=(1000,), R=5, n_lam=4, n_eps=1, M=1)
    dev = torch.device("cuda", torch.cuda.current_device())
    n = 3_000_000  # about 12 bytes per sample: more than the static scratch holds
    samples = torch.ones(n, dtype=torch.int32, device=dev)
    r_idx = torch.empty((1, 1, 1), dtype=torch.int32, device=dev)
    with pytest.raises(kvdro.KvdroError) as e:
        kvdro.kvdro_eval_grid_noalloc(1, np.array([0, n]), samples, [1000], None, len(w.r), w.r, len(w.lam), w.lam,
                                      1, w.eps[:1], 1, w.cp[:1], w.cw[:1], r_idx=r_idx)
    assert e.value.status == kvdro.KVDRO_EINVAL and "static scratch" in str(e.value)
