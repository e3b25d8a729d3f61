"""CUDA path versus the oracle on small and ragged cases, edge cases and argument errors.

Every call goes through the C ABI (the ctypes binding).  Sizes span several
warp tiles, several CTAs and several staged sample chunks, with ragged tails in
N, R and the lam grid.
"""

import os

import numpy as np
import pytest

from oracle import oracle as O
from synth import Workload, random_case, lognormal_workload_k3_n1e3
from tests.parity import RTOL, compare_full, rel_close

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402
from paper_2607_16892_gb300.runner import run  # noqa: E402

P = {"fp32": kvdro.KVDRO_FP32, "fp64": kvdro.KVDRO_FP64, "exact": kvdro.KVDRO_EXACT}


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def make(samples_per_class, L, r, lam, eps, cp, cw, L_in=None, fractiles=(0.0, 0.5, 0.9, 1.0), name="case"):
    cls = [np.asarray(c, np.int32) for c in samples_per_class]
    off = np.zeros(len(cls) + 1, np.int64)
    off[1:] = np.cumsum([c.size for c in cls])
    K = len(cls)
    return Workload(name=name, samples=np.concatenate(cls), offsets=off,
                    L=np.broadcast_to(np.asarray(L, np.int32), (K,)).copy(),
                    L_in=np.zeros(K, np.int32) if L_in is None else np.asarray(L_in, np.int32),
                    r=np.asarray(r, np.int32), lam=np.asarray(lam, np.float64), eps=np.asarray(eps, np.float64),
                    cp=np.atleast_1d(np.asarray(cp, np.float64)), cw=np.atleast_1d(np.asarray(cw, np.float64)),
                    fractiles=np.asarray(fractiles, np.float64))


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact"])
@pytest.mark.parametrize("seed", [1, 2, 3])
def test_random_ragged_cases(prec, seed):
    w = random_case(seed, K=3, N=(5000, 777, 33), L=(3000, 3000, 3000), R=45, n_lam=37, n_eps=4, M=3,
                    lam_range=(1e-3, 200.0), eps_max=300.0)
    gpu = run(w, P[prec])
    compare_full(w, gpu, O.solve(w), prec)


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact"])
def test_per_class_support_and_input_length(prec):
    w = random_case(7, K=4, N=(2100, 129, 128, 1), L=(900, 1500, 2000, 1200), L_in=(0, 50, 10, 200), R=33,
                    n_lam=16, n_eps=3, M=2, integer_costs=True)
    compare_full(w, run(w, P[prec]), O.solve(w), prec)


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact"])
def test_lognormal_k3_n1e3_full_grid(prec):
    w = lognormal_workload_k3_n1e3()
    rep = compare_full(w, run(w, P[prec]), O.solve(w), prec)
    if prec != "fp32":
        assert rep["r_idx_exact"] > 0


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact"])
def test_max_lambda_grid_and_single_points(prec):
    nl = 128 if prec == "fp64" else 256
    rng = np.random.default_rng(5)
    w = make([rng.integers(0, 500, 3000), rng.integers(200, 501, 17)], 500, [0, 250, 500],
             np.logspace(-4, 3, nl), [0.0, 40.0], [15.0, 2.0], [1.0, 0.5])
    compare_full(w, run(w, P[prec]), O.solve(w), prec)
    w1 = make([[7]], 10, [3], [0.5], [2.0], 3.0, 1.0, fractiles=[0.0, 1.0])
    compare_full(w1, run(w1, P[prec]), O.solve(w1), prec)


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact"])
def test_degenerate_inputs(prec):
    L = 64
    cases = [
        make([np.full(300, 20)], L, np.arange(0, L + 1), [0.0, 0.3, 1.0, 5.0], [0.0, 3.0], 4.0, 1.0),  # one value
        make([np.array([0, 0, L, L, 0])], L, [0, 1, 32, 63, 64], [0.0, 2.0, 9.0], [0.0, 100.0], 4.0, 1.0),  # ends
        make([np.arange(0, L + 1)], L, np.arange(0, L + 1, 7), [0.5, 2.0], [1.0], 0.0, 1.0),  # c_p = 0
        make([np.arange(0, L + 1)], L, np.arange(0, L + 1, 7), [0.5, 2.0], [1.0], 3.0, 0.0),  # c_w = 0
        make([np.arange(3, 40)], L, [10, 20, 30], [0.0], [0.0, 5.0], 2.0, 1.0),  # lam = 0 only
    ]
    for w in cases:
        compare_full(w, run(w, P[prec]), O.solve(w), prec)


def test_worked_example_values():
    import json
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "worked_example_n3_L10.json")))
    w = make([g["samples"]], g["L"], g["r"], g["lam"], g["eps"], g["cp"], g["cw"], fractiles=g["fractiles"])
    out = run(w, kvdro.KVDRO_FP64)
    np.testing.assert_allclose(out["S"][0, 0], g["S"], rtol=1e-13)
    np.testing.assert_allclose(out["cost"][0, :, 0], g["cost"], rtol=1e-13)
    assert out["lam_idx"][0, :, 0].tolist() == g["lam_idx"]
    assert out["r_idx"][0, :, 0].tolist() == g["r_idx"]
    assert out["quant"][0].tolist() == g["quant"]
    np.testing.assert_allclose(out["fhat"][0, :, 0], g["fhat"], rtol=0)


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact"])
def test_host_buffers_match_device_buffers(prec):
    w = random_case(21, K=2, N=(3000, 211), L=(700, 700), R=19, n_lam=20, n_eps=2, M=2)
    a = run(w, P[prec])
    b = run(w, P[prec], host_outputs=True)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


@pytest.mark.parametrize("prec", ["fp64", "fp32", "exact", "envelope"])
def test_host_outputs_copied_in_regime_blocks_match_device_outputs(prec):
    """With many regimes, host outputs come back in blocks of regimes on the context's copy
    stream while later blocks evaluate: 37 regimes make blocks of 3 with a ragged last one, and
    150 lam values (100 in FP64) make the exact kernel run two lam blocks per regime block."""
    w = random_case(23, K=2, N=(2500, 90), L=(900, 900), R=13, n_lam=100 if prec == "fp64" else 150, n_eps=3, M=37,
                    lam_range=(1e-3, 50.0), eps_max=200.0)
    mode = kvdro.KVDRO_ENVELOPE if prec == "envelope" else P[prec]
    a = run(w, mode)
    b = run(w, mode, host_outputs=True)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


def test_repeatable_bit_for_bit():
    w = random_case(22, K=2, N=(9000, 300), L=(2000, 2000), R=40, n_lam=50, n_eps=3, M=2)
    a = run(w, kvdro.KVDRO_FP32)
    b = run(w, kvdro.KVDRO_FP32)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


def test_reload_and_reuse_context():
    ctx = kvdro.kvdro_create(0)
    try:
        for seed in (31, 32):
            w = random_case(seed, K=2, N=(1000 + seed, 50), L=(400, 400), R=11, n_lam=9, n_eps=2, M=1)
            compare_full(w, run(w, kvdro.KVDRO_FP64, ctx=ctx), O.solve(w), "fp64")
    finally:
        kvdro.kvdro_destroy(ctx)


# ------------------------------------------------------------------ argument errors

def _loaded_ctx():
    ctx = kvdro.kvdro_create(0)
    s = torch.tensor([1, 2, 3, 4, 5], dtype=torch.int32, device="cuda")
    kvdro.kvdro_load_samples(ctx, 1, np.array([0, 5]), s, np.array([10]))
    return ctx


def _status(fn, *a, **kw):
    try:
        fn(*a, **kw)
    except kvdro.KvdroError as e:
        return e.status
    return kvdro.KVDRO_OK


def test_invalid_arguments_are_rejected_on_the_host():
    ctx = kvdro.kvdro_create(0)
    try:
        ev = lambda **kw: kvdro.kvdro_eval_grid(ctx, kvdro.KVDRO_FP32, 1, [1], 1, [1.0], 1, [0.0], 1, [2.0], [1.0], **kw)
        assert _status(ev) == kvdro.KVDRO_ESTATE  # nothing loaded yet
        s = torch.tensor([1, 2, 3], dtype=torch.int32, device="cuda")
        with pytest.raises(ValueError):  # the binding rejects K = 0 before calling the library ...
            kvdro.kvdro_load_samples(ctx, 0, np.array([0]), s, np.array([], np.int32))
        off0 = np.array([0], np.int64)  # ... and so does the C ABI on its own
        assert kvdro.load_library().kvdro_load_samples(ctx, 0, off0.ctypes.data, s.data_ptr(), None, None,
                                                       None) == kvdro.KVDRO_EINVAL
        assert _status(kvdro.kvdro_load_samples, ctx, 1, np.array([1, 3]), s, np.array([10])) == kvdro.KVDRO_EINVAL
        assert _status(kvdro.kvdro_load_samples, ctx, 2, np.array([0, 0, 3]), s, np.array([10, 10])) == kvdro.KVDRO_EINVAL
        assert _status(kvdro.kvdro_load_samples, ctx, 1, np.array([0, 3]), s, np.array([0])) == kvdro.KVDRO_EINVAL
    finally:
        kvdro.kvdro_destroy(ctx)
    ctx = _loaded_ctx()
    try:
        E = kvdro.KVDRO_EINVAL
        f = kvdro.kvdro_eval_grid
        assert _status(f, ctx, kvdro.KVDRO_FP32, 1, [11], 1, [1.0], 1, [0.0], 1, [2.0], [1.0]) == E     # r > L
        assert _status(f, ctx, kvdro.KVDRO_FP32, 1, [-1], 1, [1.0], 1, [0.0], 1, [2.0], [1.0]) == E     # r < L_in
        assert _status(f, ctx, kvdro.KVDRO_FP32, 1, [3], 1, [-1.0], 1, [0.0], 1, [2.0], [1.0]) == E     # lam < 0
        assert _status(f, ctx, kvdro.KVDRO_FP32, 1, [3], 1, [1.0], 1, [np.nan], 1, [2.0], [1.0]) == E   # eps NaN
        assert _status(f, ctx, kvdro.KVDRO_FP32, 1, [3], 1, [1.0], 1, [0.0], 1, [np.inf], [1.0]) == E   # c_p inf
        assert _status(f, ctx, kvdro.KVDRO_FP64, 1, [3], 129, np.ones(129), 1, [0.0], 1, [2.0], [1.0]) == E  # NL cap
        assert _status(f, ctx, kvdro.KVDRO_FP32, 1, [3], 257, np.ones(257), 1, [0.0], 1, [2.0], [1.0]) == E  # NL cap
        assert _status(f, ctx, 7, 1, [3], 1, [1.0], 1, [0.0], 1, [2.0], [1.0]) == E                      # precision
        q = torch.empty(2, dtype=torch.int32, device="cuda")
        assert _status(kvdro.kvdro_quantiles, ctx, 2, [0.5, 1.5], q) == E
        # the context still works after rejected calls
        out = torch.empty(1, dtype=torch.int32, device="cuda")
        kvdro.kvdro_eval_grid(ctx, kvdro.KVDRO_FP32, 1, [3], 1, [1.0], 1, [0.0], 1, [2.0], [1.0], r_idx=out)
        kvdro.kvdro_sync(ctx)
        assert out.item() == 0
    finally:
        kvdro.kvdro_destroy(ctx)


def test_out_of_range_sample_is_reported_and_unloads():
    ctx = _loaded_ctx()
    try:
        bad = torch.tensor([1, 2, 11, 4], dtype=torch.int32, device="cuda")
        assert _status(kvdro.kvdro_load_samples, ctx, 1, np.array([0, 4]), bad, np.array([10])) == kvdro.KVDRO_EINVAL
        assert "outside" in kvdro.kvdro_last_error(ctx)
        ev = lambda: kvdro.kvdro_eval_grid(ctx, kvdro.KVDRO_FP32, 1, [1], 1, [1.0], 1, [0.0], 1, [2.0], [1.0])
        assert _status(ev) == kvdro.KVDRO_ESTATE
        neg = torch.tensor([1, -2], dtype=torch.int32, device="cuda")
        assert _status(kvdro.kvdro_load_samples, ctx, 1, np.array([0, 2]), neg, np.array([10])) == kvdro.KVDRO_EINVAL
    finally:
        kvdro.kvdro_destroy(ctx)


def test_injected_allocation_failure_reports_enomem(monkeypatch):
    for n in (1, 2, 3, 5):
        monkeypatch.setenv("KVDRO_TEST_FAIL_ALLOC", str(n))
        ctx = kvdro.kvdro_create(0)
        try:
            s = torch.arange(1, 100, dtype=torch.int32, device="cuda")
            st = _status(kvdro.kvdro_load_samples, ctx, 1, np.array([0, 99]), s, np.array([200]))
            assert st == kvdro.KVDRO_ENOMEM, n
        finally:
            kvdro.kvdro_destroy(ctx)
    monkeypatch.delenv("KVDRO_TEST_FAIL_ALLOC")
    ctx = _loaded_ctx()
    kvdro.kvdro_destroy(ctx)


@pytest.mark.parametrize("prec", ["fp32", "fp64"])
def test_a_wait_that_runs_out_reports_etimeout_and_the_device_stays_usable(monkeypatch, prec):
    """Failure detection without a fault: a test hook leaves one chunk's copy unissued, so nothing
    completes that barrier; every CTA's bounded wait (about 1 ms under the hook) gives up, the CTA
    drains the copies it did issue and sets the error bit, and the call reports KVDRO_ETIMEOUT.
    Afterwards the same CUDA context evaluates correctly."""
    rng = np.random.default_rng(3)
    w = make([rng.integers(0, 900, 20000)], 1000, [10, 200, 600], [0.5, 5.0], [0.0, 10.0], 10.0, 1.0)  # 4 staged chunks in the exact kernel, 5 in the FP64 one
    monkeypatch.setenv("KVDRO_TEST_SKIP_CHUNK", "2")
    ctx = kvdro.kvdro_create(0)
    monkeypatch.delenv("KVDRO_TEST_SKIP_CHUNK")
    try:
        kvdro.kvdro_load_samples(ctx, w.K, w.offsets, torch.from_numpy(w.samples).cuda(), w.L, w.L_in)
        dt = np.float32 if prec == "fp32" else np.float64
        cost = np.empty((1, 2, 1, 3), dt)  # host output: the call waits and reads the status
        ev = lambda **kw: kvdro.kvdro_eval_grid(ctx, P[prec], 3, w.r, 2, w.lam, 2, w.eps, 1, w.cp, w.cw, **kw)
        assert _status(ev, cost=cost) == kvdro.KVDRO_ETIMEOUT
        assert "gave up waiting" in kvdro.kvdro_last_error(ctx)
        r_idx = torch.empty((1, 2, 1), dtype=torch.int32, device="cuda")  # device output: kvdro_sync reports it
        ev(r_idx=r_idx)
        assert _status(kvdro.kvdro_sync, ctx) == kvdro.KVDRO_ETIMEOUT
        assert _status(kvdro.kvdro_sync, ctx) == kvdro.KVDRO_OK  # reported once
        # modes without staged copies are unaffected by the hook
        kvdro.kvdro_eval_grid(ctx, kvdro.KVDRO_ENVELOPE, 3, w.r, 2, w.lam, 2, w.eps, 1, w.cp, w.cw, r_idx=r_idx)
        kvdro.kvdro_sync(ctx)
    finally:
        kvdro.kvdro_destroy(ctx)
    compare_full(w, run(w, P[prec]), O.solve(w), prec)  # a context without the hook, same device


def test_the_wait_hook_of_one_context_leaves_another_on_the_same_device_unaffected(monkeypatch):
    """The bounded-wait test hook travels with one context's launches: while a hooked context's
    grid kernels give up on their never-copied chunk (device outputs, so the call returns at
    once), a second context on the same device, on another stream, evaluates correctly, and the
    hooked context still reports KVDRO_ETIMEOUT."""
    rng = np.random.default_rng(4)
    w = make([rng.integers(0, 900, 20000), rng.integers(0, 1000, 9000)], 1000, np.arange(0, 1001, 37),
             np.logspace(-2, 1.5, 24), [0.0, 10.0, 90.0], [10.0, 2.0], [1.0, 1.0])
    monkeypatch.setenv("KVDRO_TEST_SKIP_CHUNK", "1")
    hooked = kvdro.kvdro_create(0)
    monkeypatch.delenv("KVDRO_TEST_SKIP_CHUNK")
    plain = kvdro.kvdro_create(0)
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    try:
        d = torch.from_numpy(w.samples).cuda()
        for ctx in (hooked, plain):
            kvdro.kvdro_load_samples(ctx, w.K, w.offsets, d, w.L, w.L_in)
        ev = lambda ctx, st, **kw: kvdro.kvdro_eval_grid(ctx, P["fp32"], R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw,
                                                         stream=st, **kw)
        ref = O.solve(w)
        for _ in range(2):
            r_dev = torch.empty((M, E, K), dtype=torch.int32, device="cuda")
            ev(hooked, s1, r_idx=r_dev)  # its CTAs now wait out their bound on stream s1
            got = {"cost": np.empty((M, E, K, R), np.float32), "lam_idx": np.empty((M, E, K, R), np.int32),
                   "r_idx": np.empty((M, E, K), np.int32), "min_cost": np.empty((M, E, K), np.float32)}
            ev(plain, s2, **got)  # host outputs: returns once they are filled
            compare_full(w, got, ref, "fp32")
            assert _status(kvdro.kvdro_sync, plain) == kvdro.KVDRO_OK
            assert _status(kvdro.kvdro_sync, hooked) == kvdro.KVDRO_ETIMEOUT
    finally:
        kvdro.kvdro_destroy(hooked)
        kvdro.kvdro_destroy(plain)


@pytest.mark.parametrize("prec", ["exact", "fp32"])
def test_lam_blocks_keep_the_lowest_index_on_ties_across_a_block_boundary(prec):
    """More than 128 lam values run as consecutive launches over blocks of 128.  Here the second
    block repeats the first block's last value (lam = 3) 128 times.  Equal lam values give
    bit-identical objectives, so a minimum reached at lam = 3 must report index 127 (at eps = 0
    with c_p = 10 most cells reach it: S does not increase in lam) and no index above 127 may
    appear; the rest matches the oracle."""
    rng = np.random.default_rng(17)
    head = np.logspace(-3, np.log10(3.0), 128)
    lam = np.concatenate([head, np.full(128, head[-1])])
    w = make([rng.integers(0, 3000, 5000), rng.integers(0, 3000, 700)], 3000, np.arange(0, 3001, 97), lam,
             [0.0, 0.5, 20.0, 400.0], [10.0, 0.7], [1.0, 2.0])
    got = run(w, P[prec])
    assert got["lam_idx"].max() <= 127
    assert (got["lam_idx"][0, 0] == 127).any()  # regime c_p = 10, eps = 0
    compare_full(w, got, O.solve(w), prec)


@pytest.mark.parametrize("prec", ["exact", "fp32"])
@pytest.mark.parametrize("nl,L", [(1, 3000), (2, 3000), (129, 3000), (130, 3000), (1, (1 << 20) + 5), (129, (1 << 20) + 5)])
def test_one_or_two_lam_values_and_blocks_ending_in_them(prec, nl, L):
    """A grid of one or two lam values -- or a block of 128 followed by one or two -- takes the
    8 r x 2 lam tiles (all-integer); a ragged r count (not a multiple of the CTA's 128 rows) and a
    support above 2^19 included."""
    rng = np.random.default_rng(nl + L % 97)
    w = make([np.concatenate([[0, L], rng.integers(0, L + 1, 4100)]), rng.integers(0, L + 1, 333)], L,
             np.unique(np.linspace(0, L, 203).round()).astype(np.int32), np.logspace(-3, 2, nl),
             [0.0, 3.0, 250.0], [10.0, 0.4], [1.0, 2.5])
    compare_full(w, run(w, P[prec]), O.solve(w), prec)


def test_exact_mode_rejects_support_above_its_limit():
    ctx = kvdro.kvdro_create(0)
    try:
        s = torch.tensor([1, 2, 3], dtype=torch.int32, device="cuda")
        kvdro.kvdro_load_samples(ctx, 1, np.array([0, 3]), s, np.array([(1 << 22) + 1]))
        ev = lambda p: kvdro.kvdro_eval_grid(ctx, p, 1, [3], 1, [1.0], 1, [0.0], 1, [2.0], [1.0])
        assert _status(ev, kvdro.KVDRO_EXACT) == kvdro.KVDRO_EINVAL
        ev(kvdro.KVDRO_FP64)  # the other modes accept it
        ev(kvdro.KVDRO_FP32)
    finally:
        kvdro.kvdro_destroy(ctx)


@pytest.mark.parametrize("prec", ["exact", "fp64", "envelope"])
def test_multipliers_and_costs_far_below_fp32_range(prec):
    """kappa below FP32's smallest normal (the FP32 estimate of a cell's threshold overflows and the
    FP64 quotient settles it), and c_w or mu many orders below c_p (the excess offset d must not
    lose them to cancellation).  FP32 outputs cannot hold costs of 1e-248; FP32 requests run the
    same exact kernel (test_fp32_results_are_the_exact_results_rounded)."""
    rng = np.random.default_rng(17)
    w = make([rng.integers(0, 300, 2000), rng.integers(100, 301, 60)], 300, [0, 7, 150, 299, 300],
             [1e-300, 1e-200, 1e-45, 1e-38, 1e-20, 0.5], [0.0, 1e-10, 3.0], [10.0, 1e-300, 2.0], [1.0, 1e-300, 1e-250])
    mode = kvdro.KVDRO_ENVELOPE if prec == "envelope" else P[prec]
    compare_full(w, run(w, mode), O.solve(w), "fp64" if prec == "envelope" else prec)


@pytest.mark.parametrize("prec", ["exact", "fp64", "envelope"])
def test_multipliers_costs_and_radii_far_above_fp32_range(prec):
    """Costs, multipliers and radii around 1e150 (their products near 1e250 stay finite in FP64)."""
    rng = np.random.default_rng(19)
    w = make([rng.integers(0, 5000, 1500), rng.integers(4000, 5001, 40)], 5000, [0, 1, 2500, 4999, 5000],
             [1e-3, 1.0, 1e120, 1e150, 3e150], [0.0, 1.0, 1e100], [1e150, 1.0, 2e150], [1.0, 1e150, 5e149])
    mode = kvdro.KVDRO_ENVELOPE if prec == "envelope" else P[prec]
    compare_full(w, run(w, mode), O.solve(w), "fp64" if prec == "envelope" else prec)


@pytest.mark.parametrize("nl", [37, 128, 129, 256])
def test_fp32_results_are_the_exact_results_rounded(nl):
    """With every support at most 2^22 an FP32 request runs the exact kernel and rounds its
    results: S, cost and the minimum cost are the FP64 exact-mode values cast to FP32, bit for bit
    (lam counts on both sides of the 128 / 256 tile variants)."""
    w = random_case(21, K=3, N=(3000, 517, 40), L=(4000, 4000, 4000), R=29, n_lam=nl, n_eps=3, M=2,
                    lam_range=(1e-3, 300.0), eps_max=500.0)
    f32, ex = run(w, P["fp32"]), run(w, P["exact"])
    for key in ("S", "cost"):
        assert np.array_equal(f32[key], ex[key].astype(np.float32)), key
    compare_full(w, ex, O.solve(w), "exact")


@pytest.mark.parametrize("prec", ["exact", "fp32"])
def test_exact_kernel_at_its_largest_support(prec):
    """L = 2^22, the largest support the exact kernel takes: its FP32 sums fold after every
    load; samples at 0 and at L, cells with every sample active (lam = 0) and none active."""
    L = 1 << 22
    rng = np.random.default_rng(12)
    w = make([np.concatenate([[0, 0, L, L], rng.integers(0, L + 1, 2500)]), rng.integers(L - 3000, L + 1, 700)], L,
             [0, 1, 1 << 21, L - 1, L], np.concatenate([[0.0], np.logspace(-3, 2, 20)]), [0.0, 5000.0], [10.0, 0.5],
             [1.0, 2.0])
    compare_full(w, run(w, P[prec]), O.solve(w), prec)


@pytest.mark.parametrize("L,nl", [(1 << 19, 40), ((1 << 19) + 1, 40), ((1 << 20) + 3, 200)])
def test_exact_variants_either_side_of_the_integer_split(L, nl):
    """Supports up to 2^19 run half of every row's columns on packed FP32 adds; above, every
    column on integer absolute differences (narrow tiles, and wide ones for 200 lam values).
    Both forms are exact."""
    rng = np.random.default_rng(41)
    w = make([np.concatenate([[0, L], rng.integers(0, L + 1, 3000)]), rng.integers(L - 9000, L + 1, 500)], L,
             [0, 1, L // 3, L - 1, L], np.logspace(-3, 2, nl), [0.0, 700.0], [10.0, 0.5], [1.0, 3.0])
    compare_full(w, run(w, kvdro.KVDRO_EXACT), O.solve(w), "exact")
    compare_full(w, run(w, kvdro.KVDRO_FP32), O.solve(w), "fp32")


def test_integer_variant_with_input_lengths_and_ragged_classes():
    """The all-integer variant (support above 2^19) with per-class input lengths, a class of 1 and
    one of 67 samples (padding in its only load), and a support point at each end."""
    L = (1 << 20) + 17
    rng = np.random.default_rng(43)
    w = make([np.concatenate([[0, L], rng.integers(0, L + 1, 2047)]), [L // 2], rng.integers(0, L + 1, 67)], L,
             [40, 41, 5000, L // 2, L], np.logspace(-2, 1.5, 29), [0.0, 3.0, 9000.0], [4.0, 1.0, 0.25],
             [1.0, 2.0, 1.0], L_in=[40, 0, 7])
    compare_full(w, run(w, kvdro.KVDRO_EXACT), O.solve(w), "exact")


@pytest.mark.parametrize("prec", ["fp32", "fp64"])
def test_staging_offsets_differ_by_class(prec):
    """A class staged as x + 2^23 (support at most 2^22) beside one staged as x (support above
    2^22) in one request: the FP32-arithmetic and FP64 kernels remove each class's own offset."""
    L_small, L_big = 3000, (1 << 22) + 100
    rng = np.random.default_rng(31)
    w = make([np.concatenate([[0, L_small], rng.integers(0, L_small + 1, 2000)]),
              np.concatenate([[0, 1, L_big], rng.integers(0, L_big + 1, 900)])],
             [L_small, L_big], [0, 1, 1500, 2999, 3000], np.logspace(-3, 2, 24), [0.0, 300.0], [10.0, 1.0],
             [1.0, 2.0])
    compare_full(w, run(w, P[prec]), O.solve(w), prec)


@pytest.mark.parametrize("nl", [40, 200])
def test_fp32_above_the_exact_limit_matches_the_oracle(nl):
    """Supports above 2^22 take the FP32-arithmetic kernel (the exact one needs L <= 2^22)."""
    L = (1 << 22) + 4096
    rng = np.random.default_rng(11)
    w = make([rng.integers(0, L + 1, 3000), np.concatenate([[0, L], rng.integers(L - 5000, L + 1, 300)])], L,
             [1, 1 << 21, L - 2, L], np.logspace(-3, 2, nl), [0.0, 1000.0], [10.0, 1.0], [1.0, 1.0])
    compare_full(w, run(w, kvdro.KVDRO_FP32), O.solve(w), "fp32")


def _random_shape_case(seed):
    """A seeded random problem: 1-4 classes of 1-2000 samples (some repeated values), a support
    from 1 to above 2^22, input lengths, 1-200 reservations, 1-256 lam values, 1-6 radii (eps = 0
    included), 1-3 regimes with a zero cost now and then."""
    rng = np.random.default_rng(1000 + seed)
    K = int(rng.integers(1, 5))
    L = int(rng.choice([1, 7, 100, 3000, 40000, (1 << 19) + 3], p=[.05, .08, .22, .35, .2, .1]))
    if seed % 8 == 7:
        L = (1 << 22) + 9  # FP32 requests take the FP32-arithmetic kernel
    # input lengths spread by at most L, so that every class shares some reservations
    L_in = int(rng.integers(0, 50)) + rng.integers(0, min(L, 50) + 1, K) if rng.random() < 0.4 else np.zeros(K, np.int64)
    cls = []
    for _ in range(K):
        n = int(rng.integers(1, 2001))
        x = rng.integers(0, L + 1, n) if rng.random() < 0.5 else np.minimum(L, rng.geometric(1.0 / max(2, L // 20), n))
        cls.append(x)
    lo, hi = int(L_in.max()), int((L_in + L).min())
    R = int(rng.integers(1, 201))
    r = np.unique(rng.integers(lo, hi + 1, R))
    NL = int(rng.integers(1, 257))
    lam = np.sort(np.concatenate([[0.0] if rng.random() < 0.2 else [], rng.uniform(0, 1, NL) ** 3 * 60]))[:NL]
    E = int(rng.integers(1, 7))
    eps = np.concatenate([[0.0], rng.uniform(0, 2 * L + 1, E - 1)])
    M = int(rng.integers(1, 4))
    cp = rng.uniform(0, 30, M) * (rng.random(M) > 0.1)
    cw = rng.uniform(0, 4, M) * (rng.random(M) > 0.1)
    return make(cls, L, r, lam, eps, cp, cw, L_in=L_in, name=f"sweep{seed}")


@pytest.mark.parametrize("seed", range(48))
def test_random_shapes_every_mode(seed):
    """Every mode the shape admits (FP32 always; exact up to a support of 2^22; FP64 up to 128 lam
    values; the envelope mode) against the oracle, on seeded random shapes."""
    w = _random_shape_case(seed)
    ref = O.solve(w)
    modes = ["fp32", "envelope"]
    if w.L.max() <= (1 << 22):
        modes.append("exact")
    if len(w.lam) <= 128:
        modes.append("fp64")
    for mode in modes:
        prec = {"fp32": kvdro.KVDRO_FP32, "fp64": kvdro.KVDRO_FP64, "exact": kvdro.KVDRO_EXACT,
                "envelope": kvdro.KVDRO_ENVELOPE}[mode]
        compare_full(w, run(w, prec), ref, "fp32" if mode == "fp32" else "fp64")


@pytest.mark.parametrize("seed", range(0, 48, 3))
def test_random_shapes_exact_dual(seed):
    """The exact dual over gamma >= 0 against the oracle's, on the same seeded random shapes."""
    from tests.test_gpu_dual import check_dual, run_dual
    w = _random_shape_case(seed)
    check_dual(w, run_dual(w), O.solve_dual(w), n_gamma=16, seed=seed)


@pytest.mark.parametrize("seed", range(1, 48, 3))
def test_random_shapes_no_allocation_entry_point(seed):
    """The allocation-free entry point against the oracle on the same shapes (those whose scratch
    fits its static array)."""
    w = _random_shape_case(seed)
    dev = torch.device("cuda", 0)
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    out = {"cost": torch.empty((M, E, K, R), dtype=torch.float32, device=dev),
           "lam_idx": torch.empty((M, E, K, R), dtype=torch.int32, device=dev),
           "r_idx": torch.empty((M, E, K), dtype=torch.int32, device=dev),
           "min_cost": torch.empty((M, E, K), dtype=torch.float32, device=dev),
           "fhat": torch.empty((M, E, K), dtype=torch.float64, device=dev)}
    try:
        kvdro.kvdro_eval_grid_noalloc(K, w.offsets, torch.from_numpy(w.samples).to(dev), w.L, w.L_in, R, w.r, NL,
                                      w.lam, E, w.eps, M, w.cp, w.cw, **out)
    except kvdro.KvdroError as e:
        if e.status == kvdro.KVDRO_EINVAL and "static scratch" in str(e):
            pytest.skip("scratch larger than the static array")
        raise
    torch.cuda.synchronize()
    compare_full(w, {k: v.cpu().numpy() for k, v in out.items()}, O.solve(w), "fp32")


def _random_large_case(seed):
    """Seeded random shapes with many staged chunks per class (up to 40,000 samples), so that the
    folds and the chunk ring turn over many times, with ragged last chunks."""
    rng = np.random.default_rng(5000 + seed)
    K = int(rng.integers(1, 5))
    L = int(rng.choice([300, 3000, 40000, 131072, (1 << 19) + 3, (1 << 21) + 1]))
    if seed % 6 == 5:
        L = (1 << 22) + 9
    cls = []
    for _ in range(K):
        n = int(rng.integers(1, 40001))
        cls.append(np.minimum(L, np.rint(np.exp(rng.normal(np.log(max(2.0, rng.uniform(1, L / 4))), 1.0, n)))).astype(np.int64))
    r = np.unique(rng.integers(0, L + 1, int(rng.integers(1, 301))))
    NL = int(rng.integers(1, 257))
    lam = np.sort(rng.uniform(0, 1, NL) ** 3 * 60)
    E = int(rng.integers(1, 7))
    eps = np.concatenate([[0.0], rng.uniform(0, 2 * L + 1, E - 1)])
    M = int(rng.integers(1, 4))
    cp = rng.uniform(0, 30, M) * (rng.random(M) > 0.1)
    cw = rng.uniform(0, 4, M) * (rng.random(M) > 0.1)
    return make(cls, L, r, lam, eps, cp, cw, name=f"large{seed}")


@pytest.mark.parametrize("seed", range(18))
def test_random_large_shapes_every_mode(seed):
    """Many chunks per class: every cell against the oracle's envelope sums (pinned against the
    direct sums), and direct per-term sums on sampled cells."""
    from tests.parity import oracle_from_S
    w = _random_large_case(seed)
    S_env = O.envelope_grid(w)
    ora = oracle_from_S(w, S_env)
    rng = np.random.default_rng(seed)
    M, K, R, NL = S_env.shape
    cells = [rng.integers(0, n, 24) for n in (M, K, R, NL)]
    direct = O.eval_cells(w, *cells)
    rel_close(S_env[tuple(cells)], direct, 1e-10, "envelope vs direct")
    modes = ["fp32"] + (["exact"] if w.L.max() <= (1 << 22) else []) + (["fp64"] if NL <= 128 else [])
    for mode in modes:
        compare_full(w, run(w, P[mode]), ora, "fp32" if mode == "fp32" else "fp64")


@pytest.mark.parametrize("L", [65534, 32767, 16382, 131070])
def test_exact_sums_stay_exact_at_the_fold_bound(L):
    """The exact kernel folds its packed FP32 sums after fe loads, fe the largest power of two with
    2 fe (L + 1) <= 2^24; each L here sits just below such a bound, so a lane's sums reach nearly
    2^24 by the fold.  Samples crowd the top of the support and the reservations its bottom (every
    |x - c| near L, odd and even), and the classes end in a large ragged chunk after one, two or
    three full ones, so the loads since the last fold do not restart at a chunk boundary.  One load
    past the bound rounds the sums: the exact mode must still meet the envelope mode (same integer
    sums, O(1) per cell) to 1e-12 and the oracle to 1e-9."""
    rng = np.random.default_rng(L)
    sizes = (12144, 3 * 6144 + 6100, 2 * 6144 + 6100, 4 * 4096 + 4000)
    cls = [L - rng.integers(0, 1 + L // 64, n) for n in sizes]
    r = np.array([0, 1, 2, 3, 7, 30, L // 2, L - 1, L])
    lam = np.array([0.01, 0.7, 1.0, 3.0, 9.5, 10.0, 25.0, 1e3])  # below, at and above c_w and c_p
    w = make(cls, L, r, lam, [0.0, 5.0, 300.0], [10.0, 1.0], [1.0, 2.0], name=f"foldbound{L}")
    ex, env = run(w, kvdro.KVDRO_EXACT), run(w, kvdro.KVDRO_ENVELOPE)
    np.testing.assert_allclose(ex["S"], env["S"], rtol=1e-12, atol=0)
    compare_full(w, ex, O.solve(w), "exact")
    compare_full(w, run(w, P["fp32"]), O.solve(w), "fp32")


@pytest.mark.parametrize("L", [900, 1 << 20, (1 << 22) + 3])
def test_class_sizes_at_chunk_and_padding_boundaries(L):
    """Classes whose sizes sit on and around the staged chunk sizes (6144 samples in the exact
    kernels, 4096 in the FP32 and FP64 ones) and the 128-sample padding unit, one sample each side:
    the fast full-chunk path, the ragged last chunk and the padded tail all meet the oracle.  The
    supports select the mixed exact kernel (900), the all-integer one (2^20) and, above 2^22, the
    FP32-arithmetic kernel for FP32 requests."""
    rng = np.random.default_rng(L)
    sizes = (1, 127, 128, 129, 4095, 4096, 4097, 6143, 6144, 6145, 12288, 12289)
    cls = [np.minimum(L, rng.integers(0, min(L, 5000) + 1, n)) for n in sizes]
    w = make(cls, L, np.unique(np.linspace(0, L, 11).astype(np.int64)), [0.02, 0.5, 1.0, 4.0, 30.0], [0.0, 7.0, 90.0],
             [6.0, 1.0], [1.0, 3.0], name=f"sizes{L}")
    ref = O.solve(w)
    modes = ["fp32", "fp64"] + (["exact"] if L <= (1 << 22) else [])
    for mode in modes:
        compare_full(w, run(w, P[mode]), ref, mode)


def test_a_wait_that_runs_out_with_regime_blocks_of_host_outputs(monkeypatch):
    """The bounded-wait test hook with several regimes and host outputs, which come back in regime
    blocks on the context's copy stream: the call still reports KVDRO_ETIMEOUT once every copy is
    done, and the device then evaluates correctly."""
    rng = np.random.default_rng(9)
    w = make([rng.integers(0, 900, 20000), rng.integers(0, 700, 3000)], 1000, [10, 200, 600], [0.5, 5.0],
             [0.0, 10.0], [10.0, 3.0, 1.5], [1.0, 1.0, 2.0])
    monkeypatch.setenv("KVDRO_TEST_SKIP_CHUNK", "1")
    ctx = kvdro.kvdro_create(0)
    monkeypatch.delenv("KVDRO_TEST_SKIP_CHUNK")
    try:
        kvdro.kvdro_load_samples(ctx, w.K, w.offsets, torch.from_numpy(w.samples).cuda(), w.L, w.L_in)
        M, E, K, R = len(w.cp), len(w.eps), w.K, len(w.r)
        out = {"cost": np.empty((M, E, K, R), np.float32), "lam_idx": np.empty((M, E, K, R), np.int32),
               "r_idx": np.empty((M, E, K), np.int32)}
        st = _status(kvdro.kvdro_eval_grid, ctx, P["fp32"], R, w.r, 2, w.lam, E, w.eps, M, w.cp, w.cw, **out)
        assert st == kvdro.KVDRO_ETIMEOUT
        assert "gave up waiting" in kvdro.kvdro_last_error(ctx)
    finally:
        kvdro.kvdro_destroy(ctx)
    compare_full(w, run(w, P["fp32"], host_outputs=True), O.solve(w), "fp32")
