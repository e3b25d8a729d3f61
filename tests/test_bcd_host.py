"""Block-coordinate descent (Alg. 1) on the host, with the oracle's worst-case cost tables.

Each block is pinned to something that does not reuse its code: brute force over Z with a
scalar objective written from eq. dro_obj / eq. capacity / eq. waiting_time, brute force over
integer reservations for LP2, closed forms for LP1 and for the M/M/1 and M/D/1 waiting times,
and the critical fractile (Prop. "Critical Fractile Structure") for the whole solve at eps = 0.
"""

import itertools
import math

import numpy as np
import pytest

pytest.importorskip("scipy")

from oracle import oracle as O  # noqa: E402
from paper_2607_16892_gb300 import bcd  # noqa: E402
from synth import CONFIGS, bcd_instance  # noqa: E402
from tests.bcd_support import oracle_tables  # noqa: E402


def small_problem(I=3, K=4, N=150, J=8, L_cap=256, **kw):
    return bcd.Problem(**bcd_instance(I, K, N, J, L_cap=L_cap, **kw))


# ---------------------------------------------------------------- the serving model

def test_config_set_is_every_budget_feasible_vector_in_lexicographic_order():
    for K, J in ((4, 8), (5, 16), (6, 12)):
        g = np.array([CONFIGS[k][0] * CONFIGS[k][1] for k in range(K)])
        want = [z for z in itertools.product(*[range(J // gk + 1) for gk in g]) if sum(a * b for a, b in zip(z, g)) <= J]
        got = bcd.config_set(g, J)
        assert got.tolist() == [list(z) for z in sorted(want)]
    # the paper's four configurations on J = 8 GPUs
    assert bcd.config_set(np.array([2, 4, 4, 8]), 8).shape == (15, 4)


def test_service_time_by_hand():
    p = small_problem(I=1, K=4)
    T = bcd.service_time(p)
    x = p.class_samples(0).astype(np.float64)
    for k in range(p.nK):
        want = (p.pp[k] * p.alpha * p.L_in[0] / p.C[k] + p.beta * x.mean() / p.B[k]
                + p.n_layers * p.tau[k] * p.t_ar)
        assert T[0, k] == pytest.approx(want, rel=1e-14)


def test_service_cv2_deterministic_and_two_point():
    p = small_problem(I=1, K=2)
    p.samples = np.full(p.samples.size, 50, np.int32)
    assert np.all(np.abs(bcd.service_cv2(p)) < 1e-12)        # every request takes the same time
    half = p.samples.size // 2
    p.samples = np.concatenate([np.full(half, 10), np.full(p.samples.size - half, 90)]).astype(np.int32)
    cv2 = bcd.service_cv2(p)
    for k in range(p.nK):
        a = p.pp[k] * p.alpha * p.L_in[0] / p.C[k] + p.n_layers * p.tau[k] * p.t_ar
        t1, t2 = a + p.beta * 10 / p.B[k], a + p.beta * 90 / p.B[k]
        n1, n2 = half, p.samples.size - half
        m = (n1 * t1 + n2 * t2) / (n1 + n2)
        var = (n1 * (t1 - m) ** 2 + n2 * (t2 - m) ** 2) / (n1 + n2)
        assert cv2[k] == pytest.approx(var / m ** 2, rel=1e-9)


@pytest.mark.parametrize("groups", [1, 3])
def test_waiting_time_reduces_to_mm1_and_md1(groups):
    """Pollaczek-Khinchin with C_s^2 = 1 is the M/M/1 queueing delay rho T / (1 - rho); with
    C_s^2 = 0 the M/D/1 one rho T / (2 (1 - rho)) (textbook results)."""
    p = small_problem(I=1, K=1)
    T = bcd.service_time(p)
    z = np.array([groups])
    pi = np.array([[1.0]])
    p.arrival = np.array([0.6 * groups / T[0, 0]])              # rho = 0.6 per group
    rho = p.arrival[0] * T[0, 0] / groups
    W1 = bcd.waiting_time(p, T, np.array([1.0]), pi, z)[0]
    W0 = bcd.waiting_time(p, T, np.array([0.0]), pi, z)[0]
    assert W1 == pytest.approx(rho * T[0, 0] / (1 - rho), rel=1e-12)
    assert W0 == pytest.approx(rho * T[0, 0] / (2 * (1 - rho)), rel=1e-12)
    p.arrival = np.array([1.01 * groups / T[0, 0]])             # overloaded: no finite wait
    assert math.isinf(bcd.waiting_time(p, T, np.array([1.0]), pi, z)[0])


# ---------------------------------------------------------------- Block 2

def test_block2_rule_as_printed():
    p = small_problem(I=2, K=3)
    T = bcd.service_time(p)
    z = np.array([2, 1, 0])
    pi = np.array([[0.5, 0.5, 0.0], [1.0, 0.0, 0.0]])
    p.arrival = np.array([6.0 / T[0, 0], 0.5 / T[1, 0]])    # u_00 pi_00 / z_0 = 1.5, u_10 pi_10 / z_0 = 0.25
    u = p.arrival[:, None] * T
    want = np.zeros((2, 3), np.int32)
    for i in range(2):
        for k in range(3):
            want[i, k] = int(z[k] > 0 and u[i, k] * pi[i, k] / z[k] > 1.0)
    assert want[0, 0] == 1 and want[1, 0] == 0 and want[:, 2].sum() == 0
    assert np.array_equal(bcd.block2(p, T, z, pi), want)


def test_block2_never_fires_where_the_waiting_time_is_finite():
    """u_ik pi_ik / z_k <= u_k, so at every point with u_k < 1 the printed rule gives delta = 0."""
    rng = np.random.default_rng(7)
    p = small_problem(I=4, K=4)
    T = bcd.service_time(p)
    for _ in range(200):
        z = rng.integers(0, 3, p.nK)
        pi = rng.random((p.I, p.nK)) * (z > 0)[None, :]
        pi /= np.maximum(pi.sum(axis=1, keepdims=True), 1.0)
        load = (p.arrival[:, None] * pi * T).sum(axis=0)
        zz = np.maximum(z, 1)
        if np.all(load / zz < 1.0):
            assert bcd.block2(p, T, z, pi).sum() == 0


# ---------------------------------------------------------------- Block 3

def scalar_objective(p, T, cv2, f, z, eta, pi, delta):
    """eq. dro_obj with eq. waiting_time, eq. slo_slack, eq. capacity and the GPU budget,
    written out with loops; inf where a constraint fails."""
    if sum(int(z[k]) * int(p.tau[k] * p.pp[k]) for k in range(p.nK)) > p.J:
        return math.inf
    W = [0.0] * p.nK
    for k in range(p.nK):
        lam_pi = sum(p.arrival[i] * pi[i, k] for i in range(p.I))
        if lam_pi == 0.0:
            continue
        if z[k] == 0:
            return math.inf
        U = sum(p.arrival[i] * pi[i, k] * T[i, k] for i in range(p.I))
        u = U / z[k]
        if u > p.u_max * (1 + 1e-9) or u >= 1.0:
            return math.inf
        W[k] = u * (1 + cv2[k]) / (2 * (1 - u)) * (U / lam_pi)
        lhs = sum((1 + p.kappa) * p.arrival[i] * T[i, k] * pi[i, k] / z[k]
                  * (p.L_in[i] + eta[i] - delta[i, k] * p.L_pre[i]) for i in range(p.I))
        lhs += sum(delta[i, k] * p.L_pre[i] for i in range(p.I))
        if lhs > p.M[k] * (1 + 1e-7):
            return math.inf
    total = 0.0
    for i in range(p.I):
        a = sum(pi[i, k] for k in range(p.nK))
        lat = sum(pi[i, k] * (W[k] + T[i, k]) for k in range(p.nK) if pi[i, k] > 0)
        s = max(0.0, lat - a * p.D[i])
        gpu = sum(pi[i, k] * p.c_gpu * p.tau[k] * p.pp[k] * T[i, k] for k in range(p.nK))
        total += p.arrival[i] * (a * f[i] + gpu + p.c_slo * s + (1 - a) * p.c_rej)
    return total


@pytest.mark.parametrize("seed,routed", [(0, (1, 1, 0, 0)), (1, (1, 0, 1, 0)), (2, (0, 1, 0, 0))])
def test_block3_is_the_argmin_over_Z(seed, routed):
    rng = np.random.default_rng(seed)
    p = small_problem(I=3, K=4, J=12, load=0.5)
    T = bcd.service_time(p)
    cv2 = bcd.service_cv2(p)
    Z = bcd.config_set(p.tau * p.pp, p.J)
    pi = rng.random((p.I, p.nK)) * np.array(routed, np.float64)[None, :]
    pi *= 0.8 / np.maximum(pi.sum(axis=1, keepdims=True), 1e-12)
    eta = rng.integers(0, 200, p.I)
    delta = np.zeros((p.I, p.nK), np.int32)
    f = rng.random(p.I) * 100
    vals = np.array([scalar_objective(p, T, cv2, f, z, eta, pi, delta) for z in Z])
    assert np.isfinite(vals).any() and not np.isfinite(vals).all()
    z_cur = Z[int(np.flatnonzero(np.isfinite(vals))[-1])]
    z_best, v_best = bcd.block3(p, T, cv2, Z, z_cur, eta, pi, delta, f)
    assert v_best == pytest.approx(vals.min(), rel=1e-12)
    assert scalar_objective(p, T, cv2, f, z_best, eta, pi, delta) == pytest.approx(vals.min(), rel=1e-12)
    # the current z is kept when it is a minimiser
    z_keep, _ = bcd.block3(p, T, cv2, Z, z_best, eta, pi, delta, f)
    assert np.array_equal(z_keep, z_best)


# ---------------------------------------------------------------- LP1

def _lp1_value(p, T, W, pi, d, z):
    s = np.maximum((pi * (W[None, :] + T - p.D[:, None])).sum(axis=1), 0.0)
    g = p.c_gpu * (p.tau * p.pp)[None, :] * T
    return float((p.arrival * ((pi * (d[:, None] + g - p.c_rej)).sum(axis=1) + p.c_slo * s)).sum())


@pytest.mark.parametrize("D,c_rej", [(1e9, 5000.0), (1e-3, 5000.0), (1e9, 1e-6)])
def test_lp1_one_class_one_configuration_closed_form(D, c_rej):
    """One class, one deployed configuration: the LP is linear in pi on [0, pi_max] (pi_max from
    admission, capacity and utilisation), so pi = pi_max when its coefficient is negative, else 0."""
    p = small_problem(I=1, K=2)
    p.D = np.array([D])
    p.c_rej = c_rej
    T = bcd.service_time(p)
    z = np.array([0, 2])
    W = np.array([0.0, 0.37])
    eta = np.array([100])
    delta = np.zeros((1, 2), np.int32)
    d = np.array([42.0])
    k = 1
    u = p.arrival[0] * T[0, k]
    cap = (p.M[k]) / ((1 + p.kappa) * u / z[k] * (p.L_in[0] + eta[0]))
    util = p.u_max * z[k] / u
    pi_max = min(1.0, cap, util)
    slope = d[0] + p.c_gpu * p.tau[k] * p.pp[k] * T[0, k] - p.c_rej + p.c_slo * max(W[k] + T[0, k] - p.D[0], 0.0)
    pi = bcd.lp1(p, T, W, z, eta, delta, d)
    assert pi[0, 0] == 0.0
    assert pi[0, 1] == pytest.approx(pi_max if slope < 0 else 0.0, abs=1e-9)


def test_lp1_matches_a_grid_search_over_two_configurations():
    p = small_problem(I=1, K=3, load=3.0)
    T = bcd.service_time(p)
    z = np.array([1, 1, 0])
    W = np.array([0.8, 2.5, 0.0])
    p.D = np.array([T[0, :2].mean() + 0.5])
    eta = np.array([60])
    delta = np.zeros((1, 3), np.int32)
    d = np.array([30.0])
    pi = bcd.lp1(p, T, W, z, eta, delta, d)
    best = math.inf
    n = 400
    u = p.arrival[0] * T[0]
    for a in range(n + 1):
        for b in range(n + 1 - a):
            q = np.array([[a / n, b / n, 0.0]])
            ok = all(u[k] * q[0, k] / z[k] <= p.u_max + 1e-12 and
                     (1 + p.kappa) * u[k] * q[0, k] / z[k] * (p.L_in[0] + eta[0]) <= p.M[k] for k in range(2))
            if ok:
                best = min(best, _lp1_value(p, T, W, q, d, z))
    got = _lp1_value(p, T, W, pi, d, z)
    assert got <= best + 1e-9 * abs(best)
    lip = p.arrival[0] * (abs(d[0]) + p.c_rej + p.c_slo * np.abs(W[:2] + T[0, :2] - p.D[0]).max()
                          + p.c_gpu * 8 * T[0].max())
    assert got >= best - 2 * lip / n


# ---------------------------------------------------------------- LP2

def _lp2_case(capacity_fraction, n_cfg=1):
    p = small_problem(I=3, K=max(n_cfg, 1), N=60, L_cap=40, load=0.5)
    p.L_in = np.array([30, 50, 20])
    tb = oracle_tables(p)
    T = bcd.service_time(p)
    z = np.ones(p.nK, np.int32)
    pi = np.full((p.I, p.nK), 1.0 / p.nK)
    delta = np.zeros((p.I, p.nK), np.int32)
    star = np.array([int(np.argmin(tb.cost[i, :p.L_max[i] + 1])) for i in range(p.I)])
    use = [(1 + p.kappa) * (p.arrival * T[:, k] * pi[:, k] * (p.L_in + star)).sum() for k in range(p.nK)]
    floor = [(1 + p.kappa) * (p.arrival * T[:, k] * pi[:, k] * p.L_in).sum() for k in range(p.nK)]
    p.M = np.array([floor[k] + capacity_fraction * (use[k] - floor[k]) for k in range(p.nK)])
    return p, tb, T, z, pi, delta, star


@pytest.mark.parametrize("frac,n_cfg", [(0.6, 1), (0.3, 1), (0.85, 2), (1.5, 1)])
def test_lp2_is_the_integer_optimum(frac, n_cfg):
    p, tb, T, z, pi, delta, star = _lp2_case(frac, n_cfg)
    w = p.arrival * pi.sum(axis=1)
    A = np.array([(1 + p.kappa) * p.arrival * T[:, k] * pi[:, k] / z[k] for k in range(p.nK)])
    best, arg = math.inf, None
    for e in itertools.product(*[range(p.L_max[i] + 1) for i in range(p.I)]):
        e = np.array(e)
        if np.all(A @ (p.L_in + e) <= p.M + 1e-9):
            v = float((w * tb.cost[np.arange(p.I), e]).sum())
            if v < best:
                best, arg = v, e
    eta = bcd.lp2(p, T, tb, z, pi, delta, np.zeros(p.I, np.int64))
    assert np.all(A @ (p.L_in + eta) <= p.M * (1 + 1e-9))
    got = float((w * tb.cost[np.arange(p.I), eta]).sum())
    assert got == pytest.approx(best, rel=1e-12, abs=1e-12)
    if frac >= 1.0:
        assert np.array_equal(eta, star)       # capacity does not bind: each class's lowest argmin


# ---------------------------------------------------------------- the whole solve

@pytest.fixture(scope="module")
def solved():
    p = small_problem(I=4, K=4, N=150, J=8, L_cap=512, load=0.9)
    tb = oracle_tables(p)
    return p, tb, bcd.solve(p, tb)


def test_solve_never_raises_the_objective(solved):
    p, tb, res = solved
    tr = np.asarray(res.trace)
    assert np.isfinite(res.objective)
    assert np.all(tr[1:] <= tr[:-1] * (1 + 1e-12) + 1e-12)
    assert res.objective < tr[0]                   # the initial point rejects everything


def test_solve_ends_blockwise_optimal(solved):
    """Prop. "Convergence": at the returned point no block improves the objective alone."""
    p, tb, res = solved
    T = bcd.service_time(p)
    cv2 = bcd.service_cv2(p)
    Z = bcd.config_set(p.tau * p.pp, p.J)
    f = tb.cost[np.arange(p.I), res.eta]
    val = scalar_objective(p, T, cv2, f, res.z, res.eta, res.pi, res.delta)
    assert val == pytest.approx(res.objective, rel=1e-12)
    vals = np.array([scalar_objective(p, T, cv2, f, z, res.eta, res.pi, res.delta) for z in Z])
    assert vals.min() >= res.objective * (1 - 1e-12)
    eta2 = bcd.lp2(p, T, tb, res.z, res.pi, res.delta, res.eta)
    f2 = tb.cost[np.arange(p.I), eta2]
    assert scalar_objective(p, T, cv2, f2, res.z, eta2, res.pi, res.delta) >= res.objective * (1 - 1e-12)
    assert np.array_equal(bcd.block2(p, T, res.z, res.pi), res.delta)
    assert np.all(res.r == p.L_in + res.eta)
    assert np.all((res.eta >= 0) & (res.eta <= p.L_max))


def test_solve_at_eps0_reserves_the_critical_fractile():
    """Prop. "Critical Fractile Structure" at eps = 0 with room to spare: every admitted class
    reserves L_in + x_(ceil(q N)) with q = c_p / (c_p + c_w)."""
    p = small_problem(I=3, K=4, N=200, J=8, L_cap=1024, load=0.5)
    p.eps = np.zeros(p.I)
    p.M = np.full(p.nK, 1e12)
    tb = oracle_tables(p)
    res = bcd.solve(p, tb)
    q = p.c_p / (p.c_p + p.c_w)
    for i in range(p.I):
        if res.pi[i].sum() > 0:
            x = np.sort(p.class_samples(i))
            assert res.eta[i] == x[O.quantile_rank(q, x.size) - 1]
    assert res.pi.sum() > 0


def test_block3_hands_an_unusable_configuration_to_a_routed_one():
    """A configuration with no KV capacity can carry no traffic (eq. capacity); starting from a
    deployment that holds two of its groups, Block 3 moves those GPUs to the routed
    configuration (fewer waits, eq. waiting_time), and the next Block 1 admits more."""
    p = small_problem(I=4, K=4, N=150, J=8, L_cap=512, load=0.9)
    p.M = p.M.copy()
    p.M[0] = 0.0
    tb = oracle_tables(p)
    res = bcd.solve(p, tb, z0=np.array([2, 1, 0, 0]))
    assert res.history[0]["z"] == [0, 2, 0, 0]
    assert res.outer_iterations >= 2
    assert np.all(res.pi[:, 0] == 0.0)
    assert res.history[1]["objective"] < res.history[0]["objective"]
    tr = np.asarray(res.trace)
    assert np.all(tr[1:] <= tr[:-1] * (1 + 1e-12) + 1e-12)
    with pytest.raises(ValueError):
        bcd.solve(p, tb, z0=np.array([5, 0, 0, 0]))
