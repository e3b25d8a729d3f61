"""Outputs stay inside their extents: every output array is placed between guard regions filled
with a known byte, and after each call the guards must be untouched, in every mode (FP32, FP64,
exact, envelope, the exact dual, quantiles, sorted samples, the allocation-free entry point),
for device and host buffers.  The values inside are checked against the oracle as well.  This
stands in for a memory checker, which is not available on the GPU pool."""

import numpy as np
import pytest

from oracle import oracle as O
from synth import random_case
from tests.parity import RTOL, check_argmin, compare_full, rel_close

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402

GUARD = 4096  # bytes on each side
FILL = 0xA5


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


class Guarded:
    """A buffer of GUARD + n + GUARD bytes filled with FILL; `view` is the middle, typed."""

    def __init__(self, shape, dtype, host):
        self.n = int(np.prod(shape)) * np.dtype(dtype).itemsize
        if host:
            self.buf = np.full(2 * GUARD + self.n, FILL, np.uint8)
            self.view = self.buf[GUARD:GUARD + self.n].view(dtype).reshape(shape)
        else:
            tdt = getattr(torch, np.dtype(dtype).name)
            self.buf = torch.full((2 * GUARD + self.n,), FILL, dtype=torch.uint8, device="cuda")
            self.view = self.buf[GUARD:GUARD + self.n].view(tdt).view(shape)

    def guards_intact(self):
        b = self.buf if isinstance(self.buf, np.ndarray) else self.buf.cpu().numpy()
        return bool((b[:GUARD] == FILL).all() and (b[GUARD + self.n:] == FILL).all())

    def values(self):
        return self.view if isinstance(self.view, np.ndarray) else self.view.cpu().numpy()


def _outputs(w, ft, host, with_S=True):
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    shapes = {"cost": ((M, E, K, R), ft), "lam_idx": ((M, E, K, R), np.int32), "r_idx": ((M, E, K), np.int32),
              "min_cost": ((M, E, K), ft), "fhat": ((M, E, K), np.float64)}
    if with_S:
        shapes["S"] = ((M, K, R, NL), ft)
    return {k: Guarded(sh, dt, host) for k, (sh, dt) in shapes.items()}


def _check_guards(bufs):
    for name, g in bufs.items():
        assert g.guards_intact(), f"{name}: a write outside its extent"


CASES = {"narrow": dict(seed=61, n_lam=37), "wide": dict(seed=62, n_lam=200), "blocks_of_few": dict(seed=63, n_lam=129)}


def _case(kind):
    c = CASES[kind]
    return random_case(c["seed"], K=3, N=(5000, 777, 33), L=(3000, 3000, 3000), R=45, n_lam=c["n_lam"], n_eps=4,
                       M=3, lam_range=(1e-3, 200.0), eps_max=300.0)


@pytest.mark.parametrize("host", [False, True], ids=["device", "host"])
@pytest.mark.parametrize("mode,kind", [("fp32", "narrow"), ("fp32", "wide"), ("exact", "narrow"),
                                       ("exact", "wide"), ("exact", "blocks_of_few"), ("fp64", "narrow"),
                                       ("envelope", "narrow")])
def test_grid_outputs_stay_inside_their_extents(mode, kind, host):
    w = _case(kind)
    prec = {"fp32": kvdro.KVDRO_FP32, "fp64": kvdro.KVDRO_FP64, "exact": kvdro.KVDRO_EXACT,
            "envelope": kvdro.KVDRO_ENVELOPE}[mode]
    ft = np.float32 if mode == "fp32" else np.float64
    M, E, K, R, NL, F = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam), len(w.fractiles)
    ctx = kvdro.kvdro_create(0)
    try:
        kvdro.kvdro_load_samples(ctx, K, w.offsets, torch.from_numpy(w.samples).cuda(), w.L, w.L_in)
        bufs = _outputs(w, ft, host)
        kvdro.kvdro_eval_grid(ctx, prec, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw,
                              **{k: g.view for k, g in bufs.items()})
        bufs["quant"] = Guarded((K, F), np.int32, host)
        kvdro.kvdro_quantiles(ctx, F, w.fractiles, bufs["quant"].view)
        bufs["sorted"] = Guarded((int(w.offsets[-1]),), np.int32, host)
        kvdro.kvdro_sorted_samples(ctx, bufs["sorted"].view)
        kvdro.kvdro_sync(ctx)
        torch.cuda.synchronize()
    finally:
        kvdro.kvdro_destroy(ctx)
    _check_guards(bufs)
    tol = "fp32" if mode == "fp32" else ("exact" if mode == "exact" else "fp64")
    compare_full(w, {k: g.values() for k, g in bufs.items()}, O.solve(w), tol)


@pytest.mark.parametrize("host", [False, True], ids=["device", "host"])
def test_dual_outputs_stay_inside_their_extents(host):
    w = _case("narrow")
    M, E, K, R = len(w.cp), len(w.eps), w.K, len(w.r)
    bufs = {"cost": Guarded((M, E, K, R), np.float64, host), "gamma": Guarded((M, E, K, R), np.float64, host),
            "r_idx": Guarded((M, E, K), np.int32, host), "min_cost": Guarded((M, E, K), np.float64, host),
            "fhat": Guarded((M, E, K), np.float64, host)}
    ctx = kvdro.kvdro_create(0)
    try:
        kvdro.kvdro_load_samples(ctx, K, w.offsets, torch.from_numpy(w.samples).cuda(), w.L, w.L_in)
        kvdro.kvdro_eval_dual(ctx, R, w.r, E, w.eps, M, w.cp, w.cw, **{k: g.view for k, g in bufs.items()})
        kvdro.kvdro_sync(ctx)
        torch.cuda.synchronize()
    finally:
        kvdro.kvdro_destroy(ctx)
    _check_guards(bufs)
    ref = O.solve_dual(w)
    rel_close(bufs["cost"].values(), ref["cost"], RTOL["fp64"], "dual cost")
    check_argmin(bufs["r_idx"].values(), ref["cost"], RTOL["fp64"], "dual r_idx")


@pytest.mark.parametrize("kind", ["narrow", "wide", "blocks_of_few"])
def test_noalloc_outputs_stay_inside_their_extents(kind):
    w = _case(kind)
    M, E, K, R, NL = len(w.cp), len(w.eps), w.K, len(w.r), len(w.lam)
    bufs = _outputs(w, np.float32, host=False, with_S=False)
    samples = torch.from_numpy(w.samples).cuda()
    kvdro.kvdro_eval_grid_noalloc(K, w.offsets, samples, w.L, w.L_in, R, w.r, NL, w.lam, E, w.eps, M, w.cp, w.cw,
                                  **{k: g.view for k, g in bufs.items()})
    torch.cuda.synchronize()
    _check_guards(bufs)
    compare_full(w, {k: g.values() for k, g in bufs.items()}, O.solve(w), "fp32")
