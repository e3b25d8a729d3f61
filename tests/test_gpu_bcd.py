"""Block-coordinate descent with the library's worst-case cost tables against the oracle's."""

import numpy as np
import pytest

pytest.importorskip("scipy")

from paper_2607_16892_gb300 import bcd  # noqa: E402
from synth import bcd_instance  # noqa: E402
from tests.bcd_support import oracle_tables  # noqa: E402

RTOL = 1e-9


@pytest.fixture(scope="module")
def both():
    # 5 classes (support sizes 8192 and 32768, so two library passes), 5 configurations, J = 16
    p = bcd.Problem(**bcd_instance(5, 5, 200, 16))
    return p, bcd.gpu_tables(p), oracle_tables(p)


@pytest.mark.gpu
def test_gpu_tables_match_the_oracle(both):
    p, g, o = both
    for i in range(p.I):
        L = int(p.L_max[i])
        a, b = g.cost[i, :L + 1], o.cost[i, :L + 1]
        assert np.all(np.isfinite(a))
        assert np.max(np.abs(a - b) / np.maximum(np.abs(b), 1e-300)) <= RTOL
        assert np.all(np.isinf(g.cost[i, L + 1:]))
        gam = g.gamma[i, :L + 1]
        assert np.all((gam >= 0) & (gam <= max(p.c_p, p.c_w)))
    assert np.array_equal(g.eta0, o.eta0)
    assert np.max(np.abs(g.d0 - o.d0) / np.abs(o.d0)) <= RTOL


@pytest.mark.gpu
def test_gpu_solve_matches_the_oracle_solve(both):
    p, g, o = both
    rg, ro = bcd.solve(p, g), bcd.solve(p, o)
    assert np.isfinite(rg.objective)
    assert rg.objective == pytest.approx(ro.objective, rel=1e-7)
    assert np.array_equal(rg.z, ro.z)
    # reservations agree, or differ only where the oracle's cost at both is a tie within tolerance
    for i in range(p.I):
        if rg.eta[i] != ro.eta[i]:
            assert o.cost[i, rg.eta[i]] == pytest.approx(o.cost[i, ro.eta[i]], rel=RTOL)
    tr = np.asarray(rg.trace)
    assert np.all(tr[1:] <= tr[:-1] * (1 + 1e-12) + 1e-12)
