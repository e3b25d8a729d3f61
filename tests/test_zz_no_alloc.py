"""kvdro_eval_grid_noalloc against kvdro_eval_grid and against the CPU oracle, through the C ABI.

The no-allocation entry point serves callers that cannot allocate device memory when they
need a reservation answer (for example a serving engine whose free memory all belongs to its
KV-cache pool).  It must give the same results as the context-based entry point, also when
the previous call left other data in its shared static scratch, and the oracle's results
within the FP32 tolerance, for every kernel it can choose (the exact kernel with packed and
integer columns up to a support of 2^19, the all-integer one up to 2^22, the FP32-arithmetic
one above).  This file is collected last so that a stop-at-first-failure run has already run
every other test.
"""

import numpy as np
import pytest

from oracle import oracle as O
from synth import Workload, random_case, lognormal_workload_k3_n1e3
from tests.parity import RTOL, check_argmin, compare_full, rel_close

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


def _classes_on(L, K, seed, n=(3000, 400)):
    """K (1 or 2) classes on the support [0, L], with samples at both ends, and a small grid.
    The static scratch holds 4 bytes per support point and class, so supports above 2^21
    take one class."""
    rng = np.random.default_rng(seed)
    cls = [np.concatenate([[0, L], rng.integers(0, L + 1, n[0])]).astype(np.int32),
           rng.integers(max(0, L - 5000), L + 1, n[1]).astype(np.int32)][:K]
    off = np.concatenate([[0], np.cumsum([c.size for c in cls])]).astype(np.int64)
    return Workload(name=f"classes_L{L}", samples=np.concatenate(cls), offsets=off,
                    L=np.full(K, L, np.int32), L_in=np.zeros(K, np.int32),
                    r=np.array([0, 1, L // 3, L - 1, L], np.int32), lam=np.logspace(-3, 2, 23),
                    eps=np.array([0.0, 700.0]), cp=np.array([10.0, 0.5]), cw=np.array([1.0, 3.0]),
                    fractiles=np.array([0.5]))


def test_noalloc_matches_the_oracle():
    """Against the CPU oracle (direct per-term sums, eps epilogue, argmin), not another GPU path."""
    w = random_case(303, K=3, N=(4100, 515, 37), L=(2500, 2500, 2500), R=41, n_lam=33, n_eps=3, M=2,
                    lam_range=(1e-3, 100.0), eps_max=200.0)
    rep = compare_full(w, _noalloc(w), O.solve(w), "fp32")
    assert rep["r_idx_exact"] > 0


@pytest.mark.parametrize("L,K", [((1 << 20) + 3, 2), ((1 << 22) + 4096, 1)])
def test_noalloc_large_supports_match_the_oracle(L, K):
    """A support in (2^19, 2^22] takes the all-integer exact kernel; one above 2^22 the
    FP32-arithmetic kernel.  Both through the static scratch, against the oracle."""
    w = _classes_on(L, K, 44 + K)
    compare_full(w, _noalloc(w), O.solve(w), "fp32")


def test_noalloc_reports_a_wait_that_runs_out(monkeypatch):
    """With the bounded-wait test hook set, every grid CTA gives up on the chunk whose copy is
    never issued; the call returns KVDRO_ETIMEOUT (its outputs are incomplete) instead of
    KVDRO_OK, and the next call without the hook is correct."""
    rng = np.random.default_rng(5)
    cls = rng.integers(0, 900, 20000).astype(np.int32)  # four staged chunks
    w = Workload(name="wait", samples=cls, offsets=np.array([0, cls.size], np.int64), L=np.array([1000], np.int32),
                 L_in=np.zeros(1, np.int32), r=np.array([10, 200, 600], np.int32), lam=np.array([0.5, 5.0]),
                 eps=np.array([0.0, 10.0]), cp=np.array([10.0]), cw=np.array([1.0]), fractiles=np.array([0.5]))
    monkeypatch.setenv("KVDRO_TEST_SKIP_CHUNK", "2")
    with pytest.raises(kvdro.KvdroError) as e:
        _noalloc(w)
    assert e.value.status == kvdro.KVDRO_ETIMEOUT and "gave up waiting" in str(e.value)
    monkeypatch.delenv("KVDRO_TEST_SKIP_CHUNK")
    compare_full(w, _noalloc(w), O.solve(w), "fp32")
