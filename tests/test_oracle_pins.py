"""Pins for the CPU oracle: each check ties it to something other than itself.

Brute-force suprema, the paper's epigraph LP and the primal transport LP solved
by scipy's HiGHS, the survival-function form of the empirical newsvendor cost,
the critical-fractile argmin, order invariants, a large-radius closed form, a
hand-worked example, and a brute-force quantile definition.
"""

import json
import math
import os

import numpy as np
import pytest

from oracle import oracle as O
from synth import Workload, random_case, lognormal_workload_k3_n1e3

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def one_class(samples, L, r, lam, eps, cp, cw, L_in=0, fractiles=(0.5,)):
    s = np.asarray(samples, np.int32)
    return Workload(name="pin", samples=s, offsets=np.array([0, s.size], np.int64),
                    L=np.array([L], np.int32), L_in=np.array([L_in], np.int32),
                    r=np.asarray(r, np.int32), lam=np.asarray(lam, np.float64),
                    eps=np.asarray(eps, np.float64), cp=np.atleast_1d(np.asarray(cp, np.float64)),
                    cw=np.atleast_1d(np.asarray(cw, np.float64)), fractiles=np.asarray(fractiles, np.float64))


def brute_sup(x, eta, lam, cp, cw, L):
    """max over every integer xi in [0, L] of the loss minus lam |xi - x|.  The objective is
    piecewise linear with kinks only at eta (convex, never a strict maximum) and at the
    integer x, so the supremum over the interval is attained on this integer grid."""
    xi = np.arange(0, L + 1, dtype=np.float64)
    loss = cp * np.maximum(xi - eta, 0.0) + cw * np.maximum(eta - xi, 0.0)
    return float(np.max(loss - lam * np.abs(xi - x)))


def survival_saa(samples, eta, cp, cw, L):
    """Empirical newsvendor cost from the empirical CDF (integer eta, integer samples):
    E(x-eta)^+ = sum_{t>=eta} (1 - F(t)),  E(eta-x)^+ = sum_{t<eta} F(t)."""
    xs = np.sort(np.asarray(samples))
    t = np.arange(0, L + 1)
    F = np.searchsorted(xs, t, side="right") / xs.size
    over = float(np.sum(1.0 - F[eta:L])) if eta < L else 0.0
    under = float(np.sum(F[:eta])) if eta > 0 else 0.0
    return cp * over + cw * under


# ----------------------------------------------------------------- P1: closed-form sup

def test_phi_equals_bruteforce_sup():
    rng = np.random.default_rng(1)
    for _ in range(3000):
        L = int(rng.integers(1, 60))
        x = int(rng.integers(0, L + 1))
        eta = float(rng.integers(-5, L + 6)) if rng.random() < 0.8 else float(rng.uniform(-3, L + 3))
        lam = float(rng.choice([0.0, rng.uniform(0, 0.5), rng.uniform(0, 40)]))
        cp, cw = float(rng.uniform(0, 30)), float(rng.uniform(0, 5))
        got = O.phi(x, eta, lam, cp, cw, L)
        want = brute_sup(x, eta, lam, cp, cw, L)
        assert abs(got - want) <= 1e-12 * max(1.0, abs(want)), (x, eta, lam, cp, cw, L, got, want)


def test_mean_sup_is_mean_of_bruteforce():
    rng = np.random.default_rng(2)
    for _ in range(200):
        L = int(rng.integers(2, 50))
        n = int(rng.integers(1, 12))
        xs = rng.integers(0, L + 1, n).astype(np.int32)
        eta, lam = float(rng.integers(0, L + 1)), float(rng.uniform(0, 20))
        cp, cw = float(rng.uniform(0.1, 30)), float(rng.uniform(0.1, 5))
        want = np.mean([brute_sup(x, eta, lam, cp, cw, L) for x in xs])
        assert abs(O.mean_sup(xs, eta, lam, cp, cw, L) - want) <= 1e-12 * max(1.0, abs(want))


def test_phi_mutants_are_caught_by_bruteforce():
    """The brute-force pin has power: plausible slips in the closed form each disagree with it."""
    def Qf(eta, xi, cp, cw):
        return cp * max(xi - eta, 0.0) + cw * max(eta - xi, 0.0)

    mutants = {
        "drop_L_candidate": lambda x, e, l, cp, cw, L: max(Qf(e, 0, cp, cw) - l * x, Qf(e, x, cp, cw)),
        "drop_0_candidate": lambda x, e, l, cp, cw, L: max(Qf(e, x, cp, cw), Qf(e, L, cp, cw) - l * (L - x)),
        "wrong_sign_lam": lambda x, e, l, cp, cw, L: max(Qf(e, 0, cp, cw) + l * x, Qf(e, x, cp, cw),
                                                        Qf(e, L, cp, cw) - l * (L - x)),
        "swapped_costs": lambda x, e, l, cp, cw, L: max(Qf(e, 0, cw, cp) - l * x, Qf(e, x, cw, cp),
                                                       Qf(e, L, cw, cp) - l * (L - x)),
        "transposed_distance": lambda x, e, l, cp, cw, L: max(Qf(e, 0, cp, cw) - l * (L - x), Qf(e, x, cp, cw),
                                                             Qf(e, L, cp, cw) - l * x),
    }
    rng = np.random.default_rng(3)
    cases = [(int(rng.integers(0, 31)), float(rng.integers(0, 31)), float(rng.uniform(0, 8)),
              float(rng.uniform(1, 20)), float(rng.uniform(0.2, 3)), 30) for _ in range(300)]
    for name, f in mutants.items():
        caught = any(abs(f(*c) - brute_sup(*c)) > 1e-9 for c in cases)
        assert caught, name
    # and the oracle itself agrees on all of them
    assert all(abs(O.phi(*c) - brute_sup(*c)) <= 1e-12 * max(1, abs(brute_sup(*c))) for c in cases)


# ----------------------------------------------------------------- LP duality pins

def _dual_lp(xs, eta, eps, cp, cw, L):
    """App. A eq. app_lp: min gamma eps + (1/N) sum theta_n over gamma >= 0, theta >= 0."""
    from scipy.optimize import linprog
    n = len(xs)
    c = np.concatenate([[eps], np.full(n, 1.0 / n)])
    A, b = [], []
    for i, x in enumerate(xs):
        def row(g):
            r_ = np.zeros(n + 1)
            r_[0] = g
            r_[1 + i] = -1.0
            return r_
        A.append(row(0.0)); b.append(-cp * (x - eta))             # theta >= c_p (x + L_in - r)
        A.append(row(0.0)); b.append(-cw * (eta - x))             # theta >= c_w (r - L_in - x)
        A.append(row(-(L - x))); b.append(-cp * (L - eta))        # theta >= c_p (L + L_in - r) - gamma (L - x)
        A.append(row(-float(x))); b.append(-cw * eta)             # theta >= c_w (r - L_in) - gamma x
    res = linprog(c, A_ub=np.array(A), b_ub=np.array(b), bounds=[(0, None)] * (n + 1), method="highs")
    assert res.status == 0
    return float(res.fun), float(res.x[0])


def _primal_lp(xs, eta, eps, cp, cw, L):
    """Worst-case expectation over the 1-Wasserstein ball around the empirical
    distribution (Sec. 2.4, eq. ambiguity), as a transport LP on integer support."""
    from scipy.optimize import linprog
    n = len(xs)
    xi = np.arange(L + 1, dtype=np.float64)
    loss = cp * np.maximum(xi - eta, 0) + cw * np.maximum(eta - xi, 0)
    nv = n * (L + 1)
    c = -np.tile(loss, n)
    A_eq = np.zeros((n, nv))
    for i in range(n):
        A_eq[i, i * (L + 1):(i + 1) * (L + 1)] = 1.0
    b_eq = np.full(n, 1.0 / n)
    A_ub = np.concatenate([np.abs(xi - x) for x in xs])[None, :]
    res = linprog(c, A_ub=A_ub, b_ub=[eps], A_eq=A_eq, b_eq=b_eq, bounds=[(0, None)] * nv, method="highs")
    assert res.status == 0
    return -float(res.fun)


def _gamma_kinks(xs, eta, cp, cw, L):
    """Candidate minimisers of the convex piecewise-linear dual in gamma: 0 and the
    crossings of each sample's affine pieces (the test's own bookkeeping)."""
    q0 = cp * max(-eta, 0) + cw * max(eta, 0)
    qL = cp * max(L - eta, 0) + cw * max(eta - L, 0)
    out = {0.0}
    for x in xs:
        qx = cp * max(x - eta, 0) + cw * max(eta - x, 0)
        if x > 0:
            out.add((q0 - qx) / x)
        if x < L:
            out.add((qL - qx) / (L - x))
        if 2 * x != L:
            out.add((q0 - qL) / (2 * x - L))
    return sorted(g for g in out if g >= 0)


def test_dual_lp_value_and_grid_bound():
    rng = np.random.default_rng(4)
    for _ in range(60):
        L = int(rng.integers(5, 40))
        n = int(rng.integers(1, 7))
        xs = rng.integers(0, L + 1, n)
        eta = int(rng.integers(0, L + 1))
        eps = float(rng.choice([0.0, rng.uniform(0, 2), rng.uniform(0, L)]))
        cp, cw = float(rng.uniform(0.5, 25)), float(rng.uniform(0.2, 4))
        v, g = _dual_lp(xs, eta, eps, cp, cw, L)
        # the oracle's objective at the LP's optimal multiplier equals the LP optimum
        w = one_class(xs, L, [eta], [g], [eps], cp, cw)
        res = O.solve(w)
        assert abs(res["cost"][0, 0, 0, 0] - v) <= 1e-7 * max(1.0, abs(v))
        # on any grid the minimum over lam is an upper bound of the LP optimum (gamma restricted)
        lam = np.sort(rng.uniform(0, 30, 9))
        w2 = one_class(xs, L, [eta], lam, [eps], cp, cw)
        assert O.solve(w2)["cost"][0, 0, 0, 0] >= v - 1e-9 * max(1.0, abs(v))


def test_primal_worst_case_equals_dual_minimum():
    """Strong duality (App. A Steps 2-5): the primal worst case over the ball equals
    min over gamma >= 0 of gamma eps + mean phi, the latter evaluated by the oracle."""
    rng = np.random.default_rng(5)
    for _ in range(25):
        L = int(rng.integers(4, 24))
        n = int(rng.integers(1, 5))
        xs = rng.integers(0, L + 1, n)
        eta = int(rng.integers(0, L + 1))
        eps = float(rng.choice([0.0, rng.uniform(0, 3), rng.uniform(0, L)]))
        cp, cw = float(rng.uniform(0.5, 25)), float(rng.uniform(0.2, 4))
        primal = _primal_lp(xs, eta, eps, cp, cw, L)
        dual, _ = _dual_lp(xs, eta, eps, cp, cw, L)
        assert abs(primal - dual) <= 1e-7 * max(1.0, abs(primal))
        kinks = _gamma_kinks(xs, eta, cp, cw, L)
        w = one_class(xs, L, [eta], kinks, [eps], cp, cw)
        assert abs(O.solve(w)["cost"][0, 0, 0, 0] - primal) <= 1e-7 * max(1.0, abs(primal))


# ----------------------------------------------------------------- closed forms and invariants

def test_saturated_multiplier_gives_empirical_cost():
    """lam >= max(c_p, c_w): moving mass never pays, so S is the empirical newsvendor cost."""
    rng = np.random.default_rng(6)
    for _ in range(100):
        L = int(rng.integers(5, 300))
        xs = rng.integers(0, L + 1, int(rng.integers(1, 40)))
        eta = int(rng.integers(0, L + 1))
        cp, cw = float(rng.uniform(0.1, 40)), float(rng.uniform(0.1, 5))
        lam = max(cp, cw) * float(rng.uniform(1.0, 3.0))
        want = survival_saa(xs, eta, cp, cw, L)
        got = O.mean_sup(xs.astype(np.int32), eta, lam, cp, cw, L)
        assert abs(got - want) <= 1e-11 * max(1.0, want)


def test_eps0_argmin_is_critical_fractile():
    """Prop. 'Critical Fractile Structure': at eps = 0 with the saturated multiplier on the
    grid, the lowest-index argmin over every integer r is x_(ceil(qN)), q = c_p/(c_p+c_w)."""
    rng = np.random.default_rng(7)
    done = 0
    while done < 40:
        L = int(rng.integers(10, 200))
        n = int(rng.integers(3, 60))
        cp, cw = int(rng.integers(1, 30)), int(rng.integers(1, 5))
        if (cp * n) % (cp + cw) == 0:
            continue  # exact plateau: two minimisers in exact arithmetic
        xs = np.clip(np.rint(np.exp(rng.normal(np.log(L / 4), 0.8, n))), 0, L).astype(np.int32)
        L_in = int(rng.integers(0, 50))
        r = np.arange(L_in, L_in + L + 1)
        lam = np.logspace(-2, np.log10(3 * max(cp, cw)), 9)
        res = O.solve(one_class(xs, L, r, lam, [0.0], float(cp), float(cw), L_in=L_in))
        counts = np.array([(xs <= v).sum() for v in range(L + 1)])
        v_star = int(np.argmax((cp + cw) * counts >= cp * n))  # smallest v with F(v) >= q, exact integers
        assert r[res["r_idx"][0, 0, 0]] - L_in == v_star
        done += 1


def test_cost_monotone_in_eps_and_above_empirical_cost():
    w = random_case(11, K=3, N=(300, 41, 7), L=(400, 400, 400), R=29, n_lam=17, n_eps=6, M=3, eps_max=500)
    res = O.solve(w)
    cost, S = res["cost"], res["S"]
    assert np.all(np.diff(cost, axis=1) >= 0)                     # per cell, bit-for-bit
    assert np.all(np.diff(res["min_cost"], axis=1) >= 0)
    for m in range(len(w.cp)):
        for k in range(w.K):
            for i, r in enumerate(w.r):
                saa = survival_saa(w.class_samples(k), int(r - w.L_in[k]), w.cp[m], w.cw[m], int(w.L[k]))
                assert np.all(S[m, k, i] >= saa - 1e-9 * saa)
                assert np.all(cost[m, :, k, i] >= saa - 1e-9 * saa)


def test_eps0_min_over_grid_is_empirical_cost():
    """With lam_max >= max(c_p, c_w) on the grid and eps = 0 the minimum over lam is the
    empirical cost (S is non-increasing in lam and saturates)."""
    w = random_case(12, K=2, N=(150, 33), L=(250, 250), R=19, n_lam=13, n_eps=2, M=2, lam_range=(1e-3, 500.0))
    res = O.solve(w)
    for m in range(2):
        for k in range(2):
            for i, r in enumerate(w.r):
                saa = survival_saa(w.class_samples(k), int(r - w.L_in[k]), w.cp[m], w.cw[m], int(w.L[k]))
                assert abs(res["cost"][m, 0, k, i] - saa) <= 1e-11 * max(1, saa)
                assert np.all(np.diff(res["S"][m, k, i]) <= 1e-12 * saa)


def test_large_radius_closed_form():
    """eps >= L: the ball holds every distribution on [0, L], so the worst case is
    max(Q(eta,0), Q(eta,L)); the grid value lies within lam_min * eps above it."""
    rng = np.random.default_rng(8)
    for _ in range(50):
        L = int(rng.integers(5, 500))
        xs = rng.integers(0, L + 1, int(rng.integers(1, 30)))
        eta = int(rng.integers(0, L + 1))
        cp, cw = float(rng.uniform(0.1, 40)), float(rng.uniform(0.1, 5))
        eps = float(L * rng.uniform(1, 3))
        lam = np.logspace(-6, 2, 20)
        c = O.solve(one_class(xs, L, [eta], lam, [eps], cp, cw))["cost"][0, 0, 0, 0]
        exact = max(cw * eta, cp * (L - eta))
        assert exact - 1e-9 * exact <= c <= exact + lam[0] * eps + 1e-9 * exact


# ----------------------------------------------------------------- envelope regrouping

def test_envelope_equals_bruteforce_sum():
    rng = np.random.default_rng(9)
    for _ in range(200):
        L = int(rng.integers(2, 60))
        xs = rng.integers(0, L + 1, int(rng.integers(1, 20))).astype(np.int32)
        eta = int(rng.integers(0, L + 1)) if rng.random() < 0.7 else int(rng.integers(-10, L + 10))
        lam, cp, cw = float(rng.uniform(0, 30)), float(rng.uniform(0, 30)), float(rng.uniform(0, 5))
        w = one_class(xs, L, [max(eta, 0)], [lam], [0.0], cp, cw, L_in=max(0, -eta) if eta < 0 else 0)
        got = O.envelope_grid(w)[0, 0, 0, 0]
        e = max(eta, 0) - w.L_in[0]
        want = np.mean([brute_sup(x, e, lam, cp, cw, L) for x in xs])
        assert abs(got - want) <= 1e-11 * max(1.0, abs(want))


def test_envelope_equals_direct_on_small_workload():
    w = lognormal_workload_k3_n1e3()
    S1 = O.eval_grid(w)
    S2 = O.envelope_grid(w)
    assert np.max(np.abs(S1 - S2) / np.abs(S1)) < 1e-12


# ----------------------------------------------------------------- quantiles and Fhat

def test_quantiles_match_bruteforce_definition():
    rng = np.random.default_rng(10)
    for _ in range(50):
        n = int(rng.integers(1, 200))
        xs = rng.integers(1, 500, n).astype(np.int32)
        fr = np.concatenate([[0.0, 1.0], rng.uniform(0, 1, 10), [k / n for k in range(0, n + 1, max(1, n // 7))]])
        w = one_class(xs, 500, [1], [1.0], [0.0], 1.0, 1.0, fractiles=fr)
        got = O.quantiles(w, fr)[0]
        for f, q in enumerate(fr):
            if q == 0.0:
                want = xs.min()
            else:
                want = min(v for v in np.unique(xs) if (xs <= v).sum() >= q * n)
            assert got[f] == want, (q, n)


def test_fhat_is_empirical_cdf_at_rstar():
    w = random_case(13, K=3, N=(120, 60, 9), L=(300, 300, 300), R=23, n_lam=9, n_eps=3, M=2)
    res = O.solve(w)
    for m in range(2):
        for e in range(3):
            for k in range(3):
                r = w.r[res["r_idx"][m, e, k]] - w.L_in[k]
                assert res["fhat"][m, e, k] == np.mean(w.class_samples(k) <= r)


# ----------------------------------------------------------------- hand-worked example

def test_hand_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "worked_example_n3_L10.json")))
    w = one_class(g["samples"], g["L"], g["r"], g["lam"], g["eps"], g["cp"], g["cw"], L_in=g["L_in"],
                  fractiles=g["fractiles"])
    res = O.solve(w)
    np.testing.assert_allclose(res["S"][0, 0], np.array(g["S"]), rtol=1e-14)
    np.testing.assert_allclose(res["cost"][0, :, 0], np.array(g["cost"]), rtol=1e-14)
    assert res["lam_idx"][0, :, 0].tolist() == g["lam_idx"]
    assert res["r_idx"][0, :, 0].tolist() == g["r_idx"]
    np.testing.assert_allclose(res["min_cost"][0, :, 0], g["min_cost"], rtol=1e-14)
    assert res["quant"][0].tolist() == g["quant"]
    np.testing.assert_allclose(res["fhat"][0, :, 0], g["fhat"], rtol=1e-15)
    for j, lam in enumerate(g["lam"]):
        for n, x in enumerate(g["samples"]):
            assert O.phi(x, 2.0, lam, g["cp"], g["cw"], g["L"]) == g["phi_eta2"][j][n]


def test_quantile_rank_convention():
    assert O.quantile_rank(0.0, 10) == 1
    assert O.quantile_rank(1.0, 10) == 10
    assert O.quantile_rank(0.95, 20) == 19
    assert O.quantile_rank(0.951, 20) == 20
    assert O.quantile_rank(1.0 / 3.0, 3) == 1
    assert math.isclose(20.0 / 21.0, O.quantile_rank(20.0 / 21.0, 21) / 21.0)


# ----------------------------------------------------------------- the exact dual (no lam grid)

def test_exact_dual_equals_the_paper_lp_and_the_primal_worst_case():
    rng = np.random.default_rng(14)
    for _ in range(40):
        L = int(rng.integers(4, 30))
        n = int(rng.integers(1, 6))
        xs = rng.integers(0, L + 1, n)
        eta = int(rng.integers(0, L + 1))
        eps = float(rng.choice([0.0, rng.uniform(0, 3), rng.uniform(0, L)]))
        cp, cw = float(rng.uniform(0.5, 25)), float(rng.uniform(0.2, 4))
        w = one_class(xs, L, [eta], [1.0], [eps], cp, cw)
        got = O.solve_dual(w)["cost"][0, 0, 0, 0]
        lp, _ = _dual_lp(xs, eta, eps, cp, cw, L)
        assert abs(got - lp) <= 1e-7 * max(1.0, abs(lp))
        if L <= 20:
            assert abs(got - _primal_lp(xs, eta, eps, cp, cw, L)) <= 1e-7 * max(1.0, abs(lp))


def test_exact_dual_closed_forms_and_grid_bound():
    w = random_case(15, K=2, N=(400, 23), L=(300, 300), R=13, n_lam=24, n_eps=4, M=2, eps_max=250.0,
                    lam_range=(1e-3, 300.0))
    w.eps = np.array([0.0, 3.0, 60.0, 400.0])  # the last radius exceeds L
    d = O.solve_dual(w)
    g = O.solve(w)
    assert np.all(d["cost"] <= g["cost"] * (1 + 1e-12) + 1e-12)        # the grid restricts gamma
    for m in range(2):
        for k in range(2):
            for i, r in enumerate(w.r):
                eta = int(r - w.L_in[k])
                saa = survival_saa(w.class_samples(k), eta, w.cp[m], w.cw[m], int(w.L[k]))
                assert abs(d["cost"][m, 0, k, i] - saa) <= 1e-11 * max(1.0, saa)                # eps = 0
                worst = max(w.cw[m] * eta, w.cp[m] * (int(w.L[k]) - eta))
                assert abs(d["cost"][m, 3, k, i] - worst) <= 1e-11 * max(1.0, worst)           # eps >= L
    assert np.all(np.diff(d["cost"], axis=1) >= -1e-9)                                        # monotone in eps
