"""Block-coordinate descent over configuration, routing, caching and reservation (Alg. 1).

The joint problem of Sec. 3 (eq. dro_obj with the GPU budget, routing, capacity and SLO
constraints) is solved by the three blocks of Alg. 1 "BCD-DRO":

  Block 1  alternate LP1 (routing pi and SLO slack s for fixed reservations) and LP2
           (reservations r for fixed routing) until neither changes;
  Block 2  the prefix-caching rule delta_ik = 1[u_ik pi_ik / z_k > 1];
  Block 3  z = argmin over the configuration set
           Z = {z in Z_+^|K| : sum_k z_k tau_k p_k <= J} of the objective;

stopping when (z, delta) repeats.  The worst-case expected reservation cost of class i at
reservation r_i = L_in^i + eta, f_i(eta) = min_{gamma >= 0} gamma eps_i + S_i(eta, gamma)
(App. A, eq. app_kantorovich; the gamma and theta of LP2 eliminated exactly), is read from
a table over every integer eta in [0, L_max^i] that one ``kvdro_eval_dual`` call computes
on the GPU (``gpu_tables``); the initial point's cost at gamma = c_p comes from one
``kvdro_eval_grid`` call in ENVELOPE mode.  The rest is small host work: two HiGHS
programs (scipy) per Block 1 round and a vectorised enumeration of Z.

Readings where the paper leaves a choice open (each is also listed in the design notes):
  * r is an integer token count, so LP2 is solved exactly over integers: a MILP over the
    convex piecewise-linear cost curve, which reduces to each class's unconstrained
    argmin whenever that point satisfies every capacity constraint.
  * The waiting time W_k (eq. waiting_time) is not linear in pi; LP1 holds it at the
    value of the routing it starts from (zero routing before the first LP1) and Block 1
    recomputes it after every LP1.  LP1 also bounds every group's utilisation by u_max
    (default 0.95) so that W_k stays finite.
  * C_slo = c_slo s_i (eq. slo_slack); C_gpu and C_rej as in eq. cost.
  * The mean service time of a configuration is the arrival-weighted mean of the T_ik
    routed to it; the squared coefficient of variation C_s,k^2 is that of the service time
    of the arrival-weighted sample mix, computed once from the samples and held fixed.
  * z^(0) deploys one group of every configuration in ascending order of GPUs per group,
    round after round, until the budget is spent; pi^(0) = 0; r^(0) = L_in + E[xi] rounded to the nearest integer; gamma^(0) = c_p.
  * Ties: Block 3 keeps the current z when it attains the minimum, else takes the first
    minimiser in the lexicographic order of Z.
"""

from __future__ import annotations

import dataclasses
import json
import time
from typing import Dict, List, Optional

import numpy as np

__all__ = ["Problem", "Tables", "BcdResult", "service_time", "service_cv2", "config_set", "waiting_time",
           "objective", "lp1", "lp2", "block2", "block3", "solve", "gpu_tables"]


@dataclasses.dataclass
class Problem:
    """One instance of the joint problem (Sec. 3.1-3.4).  Arrays over classes have length I,
    arrays over configurations length nK."""

    # request classes
    arrival: np.ndarray   # lambda_i, requests per second
    L_in: np.ndarray      # input length, tokens (int)
    L_pre: np.ndarray     # cacheable shared prefix, tokens (int)
    D: np.ndarray         # latency SLO, seconds
    L_max: np.ndarray     # maximum output length, tokens (int); support of xi is [0, L_max]
    samples: np.ndarray   # int32 output-length samples, classes concatenated
    offsets: np.ndarray   # int64 [I + 1]
    eps: np.ndarray       # Wasserstein radius per class, tokens
    # configurations and cluster
    J: int                # GPU budget
    tau: np.ndarray       # tensor-parallel degree (int)
    pp: np.ndarray        # pipeline-parallel degree (int)
    M: np.ndarray         # KV-cache capacity of one serving group, tokens
    C: np.ndarray         # effective compute of one group, FLOP/s
    B: np.ndarray         # effective bandwidth of one group, bytes/s
    alpha: float          # prefill work per input token (FLOP)
    beta: float           # decode traffic per output token (bytes)
    n_layers: int         # N_L
    t_ar: float           # all-reduce latency, seconds
    # cost weights (Sec. 5.1 "System Configuration")
    c_p: float = 10.0
    c_w: float = 1.0
    c_gpu: float = 1.0
    c_slo: float = 5.0
    c_rej: float = 5000.0
    kappa: float = 0.2
    u_max: float = 0.95
    name: str = ""

    @property
    def I(self) -> int:  # noqa: E743 (the paper's symbol)
        return int(self.offsets.shape[0] - 1)

    @property
    def nK(self) -> int:
        return int(self.tau.shape[0])

    def class_samples(self, i: int) -> np.ndarray:
        return self.samples[self.offsets[i]:self.offsets[i + 1]]

    def mean_output(self) -> np.ndarray:
        return np.array([self.class_samples(i).mean() for i in range(self.I)], np.float64)


@dataclasses.dataclass
class Tables:
    """Worst-case cost curves: cost[i, eta] = f_i(eta) for eta = 0..L_max^i (inf beyond),
    a minimising gamma beside it, and the initial point (eta0, its cost at gamma = c_p)."""

    cost: np.ndarray
    gamma: np.ndarray
    eta0: np.ndarray
    d0: np.ndarray
    seconds: float = 0.0


@dataclasses.dataclass
class BcdResult:
    z: np.ndarray
    r: np.ndarray          # reservation per class, tokens (L_in + eta)
    eta: np.ndarray
    gamma: np.ndarray      # minimising gamma at each class's reservation
    pi: np.ndarray         # [I, nK]
    delta: np.ndarray      # [I, nK] int
    s: np.ndarray          # SLO slack per class
    W: np.ndarray          # waiting time per configuration
    objective: float
    parts: Dict[str, float]
    outer_iterations: int
    lp_rounds: int
    history: List[dict]
    seconds: Dict[str, float]

    def to_json(self) -> dict:
        return {"z": self.z.tolist(), "r": self.r.tolist(), "gamma": self.gamma.round(9).tolist(),
                "pi": self.pi.round(9).tolist(), "delta": self.delta.tolist(), "objective": self.objective,
                "parts": self.parts, "outer_iterations": self.outer_iterations, "lp_rounds": self.lp_rounds,
                "seconds": self.seconds}


# ---------------------------------------------------------------- the serving model (Sec. 3.1, 3.4)

def service_time(p: Problem) -> np.ndarray:
    """T[i, k] = p_k alpha L_in^i / C_k + beta E[xi_i] / B_k + N_L tau_k t_ar (eq. service_time)."""
    mean = p.mean_output()
    return (p.pp[None, :] * p.alpha * p.L_in[:, None] / p.C[None, :]
            + p.beta * mean[:, None] / p.B[None, :]
            + p.n_layers * p.tau[None, :] * p.t_ar)


def service_cv2(p: Problem) -> np.ndarray:
    """C_s,k^2: squared coefficient of variation of the per-request service time on
    configuration k over the arrival-weighted mix of every class's samples (xi in place of
    E[xi] in eq. service_time).  Fixed for the whole solve."""
    out = np.empty(p.nK)
    for k in range(p.nK):
        mom1 = mom2 = wsum = 0.0
        for i in range(p.I):
            x = p.class_samples(i).astype(np.float64)
            t = (p.pp[k] * p.alpha * p.L_in[i] / p.C[k] + p.beta * x / p.B[k] + p.n_layers * p.tau[k] * p.t_ar)
            w = p.arrival[i]
            mom1 += w * t.mean()
            mom2 += w * (t * t).mean()
            wsum += w
        m1, m2 = mom1 / wsum, mom2 / wsum
        out[k] = max(m2 - m1 * m1, 0.0) / (m1 * m1)
    return out


def config_set(gpus_per_group: np.ndarray, J: int) -> np.ndarray:
    """Every z in Z_+^nK with sum_k z_k g_k <= J, in lexicographic order (Sec. 4.3).  Built one
    configuration at a time: each partial vector is repeated once per count its remaining
    budget allows, the counts ascending."""
    g = np.asarray(gpus_per_group, np.int64)
    rows = np.zeros((1, 0), np.int32)
    left = np.array([int(J)], np.int64)
    for gk in g:
        counts = left // int(gk) + 1
        rep = np.repeat(np.arange(rows.shape[0]), counts)
        starts = np.repeat(np.cumsum(counts) - counts, counts)
        zk = (np.arange(rep.size) - starts).astype(np.int64)
        rows = np.concatenate([rows[rep], zk[:, None].astype(np.int32)], axis=1)
        left = left[rep] - zk * int(gk)
    return rows


def waiting_time(p: Problem, T: np.ndarray, cv2: np.ndarray, pi: np.ndarray, z: np.ndarray) -> np.ndarray:
    """W_k = u_k (1 + C_s,k^2) / (2 (1 - u_k)) Tbar_k with u_k = sum_i lambda_i pi_ik T_ik / z_k
    (eq. waiting_time).  0 where nothing is routed; inf where u_k >= 1 or z_k = 0 with load."""
    load = (p.arrival[:, None] * pi * T).sum(axis=0)           # sum_i lambda_i pi_ik T_ik
    rate = (p.arrival[:, None] * pi).sum(axis=0)
    W = np.zeros(p.nK)
    for k in range(p.nK):
        if rate[k] <= 0.0:
            continue
        if z[k] <= 0:
            W[k] = np.inf
            continue
        u = load[k] / z[k]
        if u >= 1.0:
            W[k] = np.inf
            continue
        W[k] = u * (1.0 + cv2[k]) / (2.0 * (1.0 - u)) * (load[k] / rate[k])
    return W


def _reservation(p: Problem, eta: np.ndarray) -> np.ndarray:
    return p.L_in.astype(np.float64) + eta.astype(np.float64)


def capacity_rows(p: Problem, T: np.ndarray, z: np.ndarray, pi: np.ndarray, delta: np.ndarray,
                  eta: np.ndarray) -> np.ndarray:
    """Left side minus right side of eq. capacity for every configuration with z_k > 0
    (<= 0 when it holds); nan where z_k = 0."""
    u = p.arrival[:, None] * T
    r_t = _reservation(p, eta)[:, None] - delta * p.L_pre[:, None]
    out = np.full(p.nK, np.nan)
    for k in range(p.nK):
        if z[k] > 0:
            out[k] = ((1.0 + p.kappa) * (u[:, k] * pi[:, k] / z[k] * r_t[:, k]).sum()
                      + (delta[:, k] * p.L_pre).sum() - p.M[k])
    return out


def objective(p: Problem, T: np.ndarray, cv2: np.ndarray, tables: Tables, z: np.ndarray, eta: np.ndarray,
              pi: np.ndarray, delta: np.ndarray, d: Optional[np.ndarray] = None, check: bool = True):
    """The objective of eq. dro_obj, sum_i lambda_i [a_i f_i(r_i) + C_gpu + C_slo + C_rej],
    and its parts; inf when a constraint (routing consistency, GPU budget, utilisation,
    capacity) fails.  ``d`` overrides f_i(r_i) (the initial point's gamma = c_p cost)."""
    if d is None:
        d = tables.cost[np.arange(p.I), eta]
    a = pi.sum(axis=1)
    W = waiting_time(p, T, cv2, pi, z)
    with np.errstate(invalid="ignore"):
        lat = np.where(pi > 0, pi * (W[None, :] + T), 0.0).sum(axis=1)
    s = np.maximum(lat - a * p.D, 0.0)
    gpu = (pi * p.c_gpu * (p.tau * p.pp)[None, :] * T).sum(axis=1)
    parts = {"dro": float((p.arrival * a * d).sum()), "gpu": float((p.arrival * gpu).sum()),
             "slo": float((p.arrival * p.c_slo * s).sum()), "rej": float((p.arrival * (1.0 - a) * p.c_rej).sum())}
    total = sum(parts.values())
    if check:
        feasible = int((z * p.tau * p.pp).sum()) <= p.J and np.all(np.isfinite(W))
        feasible = feasible and not np.any((pi.sum(axis=0) > 0) & (z <= 0))
        util = (p.arrival[:, None] * pi * T).sum(axis=0)
        feasible = feasible and np.all(util <= p.u_max * np.maximum(z, 0) * (1 + 1e-9) + 1e-12)
        cap = capacity_rows(p, T, z, pi, delta, eta)
        feasible = feasible and np.all(np.nan_to_num(cap, nan=-1.0) <= 1e-7 * np.maximum(p.M, 1.0))
        if not feasible:
            total = np.inf
    return total, parts, s, W


# ---------------------------------------------------------------- Block 1

def lp1(p: Problem, T: np.ndarray, W: np.ndarray, z: np.ndarray, eta: np.ndarray, delta: np.ndarray,
        d: np.ndarray):
    """Routing for fixed reservations, caching and configuration (Alg. 1 Block 1, LP1):
    minimise sum_i lambda_i [sum_k pi_ik (d_i + c_gpu tau_k p_k T_ik - c_rej) + c_slo s_i]
    subject to sum_k pi_ik <= 1 (eq. routing_prob), pi_ik = 0 where z_k = 0
    (eq. routing_consist), eq. capacity, the utilisation bound, and eq. slo_slack with W_k
    held fixed.  Returns pi [I, nK]."""
    from scipy.optimize import linprog

    I, nK = p.I, p.nK
    act = np.flatnonzero(z > 0)
    nA = act.size
    pi = np.zeros((I, nK))
    if nA == 0:
        return pi
    nv = I * nA + I
    c = np.zeros(nv)
    g = p.c_gpu * (p.tau * p.pp)[None, :] * T
    for i in range(I):
        for j, k in enumerate(act):
            c[i * nA + j] = p.arrival[i] * (d[i] + g[i, k] - p.c_rej)
        c[I * nA + i] = p.arrival[i] * p.c_slo
    rows, rhs = [], []
    for i in range(I):                                          # admission
        row = np.zeros(nv)
        row[i * nA:(i + 1) * nA] = 1.0
        rows.append(row)
        rhs.append(1.0)
    u = p.arrival[:, None] * T
    r_t = _reservation(p, eta)[:, None] - delta * p.L_pre[:, None]
    for j, k in enumerate(act):                                 # capacity and utilisation
        row = np.zeros(nv)
        for i in range(I):
            row[i * nA + j] = (1.0 + p.kappa) * u[i, k] / z[k] * r_t[i, k]
        rows.append(row)
        rhs.append(p.M[k] - float((delta[:, k] * p.L_pre).sum()))
        row = np.zeros(nv)
        for i in range(I):
            row[i * nA + j] = u[i, k] / z[k]
        rows.append(row)
        rhs.append(p.u_max)
    for i in range(I):                                          # SLO slack
        row = np.zeros(nv)
        for j, k in enumerate(act):
            row[i * nA + j] = W[k] + T[i, k] - p.D[i]
        row[I * nA + i] = -1.0
        rows.append(row)
        rhs.append(0.0)
    bounds = [(0.0, 1.0)] * (I * nA) + [(0.0, None)] * I
    res = linprog(c, A_ub=np.asarray(rows), b_ub=np.asarray(rhs), bounds=bounds, method="highs")
    if res.status != 0:
        raise RuntimeError(f"LP1 failed: {res.message}")
    x = np.clip(res.x[:I * nA].reshape(I, nA), 0.0, 1.0)
    x[x < 1e-12] = 0.0
    pi[:, act] = x
    return pi


def lp2(p: Problem, T: np.ndarray, tables: Tables, z: np.ndarray, pi: np.ndarray, delta: np.ndarray,
        eta_cur: np.ndarray) -> np.ndarray:
    """Reservations for fixed routing (Alg. 1 Block 1, LP2): minimise
    sum_i lambda_i a_i f_i(eta_i) over integer eta_i in [0, L_max^i] subject to eq. capacity.
    Each f_i is convex, so a class never goes above its unconstrained (lowest) argmin; when
    those argmins meet every capacity constraint they are the answer, otherwise a MILP over
    the epigraph of the piecewise-linear f_i on [0, argmin] gives the exact integer optimum."""
    I = p.I
    f = tables.cost
    star = np.array([int(np.argmin(f[i, :p.L_max[i] + 1])) for i in range(I)], np.int64)
    a = pi.sum(axis=1)
    w = p.arrival * a
    act = np.flatnonzero(z > 0)
    u = p.arrival[:, None] * T
    A = np.zeros((act.size, I))
    b = np.zeros(act.size)
    for j, k in enumerate(act):
        A[j] = (1.0 + p.kappa) * u[:, k] * pi[:, k] / z[k]
        b[j] = (p.M[k] - float((delta[:, k] * p.L_pre).sum())
                - float((A[j] * (p.L_in - delta[:, k] * p.L_pre)).sum()))
    tol = 1e-9 * np.maximum(np.abs(b), 1.0)
    if act.size == 0 or np.all(A @ star <= b + tol):
        return star
    from scipy.optimize import Bounds, LinearConstraint, milp
    from scipy.sparse import coo_matrix

    coupled = np.flatnonzero(w > 0)
    eta = star.copy()
    nc = coupled.size
    hi = np.array([max(int(star[i]), int(eta_cur[i])) for i in coupled], np.int64)
    # variables: eta_c (nc, integer), t_c (nc, continuous)
    rr, cc, vv, lo_rows, up_rows = [], [], [], [], []
    nrow = 0
    for q, i in enumerate(coupled):
        fi = f[i, :hi[q] + 1]
        for j in range(hi[q]):                                  # t_q >= f(j) + (f(j+1) - f(j)) (eta - j)
            sl = fi[j + 1] - fi[j]
            rr += [nrow, nrow]
            cc += [q, nc + q]
            vv += [sl, -1.0]
            lo_rows.append(-np.inf)
            up_rows.append(sl * j - fi[j])
            nrow += 1
        if hi[q] == 0:                                          # t_q >= f(0)
            rr.append(nrow)
            cc.append(nc + q)
            vv.append(-1.0)
            lo_rows.append(-np.inf)
            up_rows.append(-fi[0])
            nrow += 1
    for j in range(act.size):                                   # capacity
        for q, i in enumerate(coupled):
            if A[j, i] != 0.0:
                rr.append(nrow)
                cc.append(q)
                vv.append(A[j, i])
        lo_rows.append(-np.inf)
        up_rows.append(b[j])                                    # uncoupled classes have A[j, i] = 0
        nrow += 1
    Amat = coo_matrix((vv, (rr, cc)), shape=(nrow, 2 * nc)).tocsr()
    cvec = np.concatenate([np.zeros(nc), w[coupled]])
    integrality = np.concatenate([np.ones(nc), np.zeros(nc)])
    bounds = Bounds(np.concatenate([np.zeros(nc), np.full(nc, -np.inf)]),
                    np.concatenate([hi.astype(np.float64), np.full(nc, np.inf)]))
    res = milp(cvec, constraints=LinearConstraint(Amat, np.asarray(lo_rows), np.asarray(up_rows)),
               integrality=integrality, bounds=bounds, options={"mip_rel_gap": 0.0})
    if res.status != 0 or res.x is None:
        raise RuntimeError(f"LP2 failed: {res.message}")
    eta[coupled] = np.rint(res.x[:nc]).astype(np.int64)
    return eta


# ---------------------------------------------------------------- Blocks 2 and 3

def block2(p: Problem, T: np.ndarray, z: np.ndarray, pi: np.ndarray) -> np.ndarray:
    """delta_ik = 1[u_ik pi_ik / z_k > 1] with u_ik = lambda_i T_ik (Alg. 1 Block 2); 0 where z_k = 0."""
    u = p.arrival[:, None] * T
    zz = np.where(z > 0, z, 1)[None, :]
    return ((u * pi / zz > 1.0) & (z[None, :] > 0)).astype(np.int32)


def block3(p: Problem, T: np.ndarray, cv2: np.ndarray, Z: np.ndarray, z_cur: np.ndarray, eta: np.ndarray,
           pi: np.ndarray, delta: np.ndarray, d: np.ndarray, chunk: int = 131072):
    """z = argmin over Z of the objective with (r, pi, delta) fixed (Alg. 1 Block 3), every z
    evaluated.  With pi fixed, configuration k's feasibility (routing consistency, utilisation,
    eq. capacity) and waiting time depend on z_k alone, so they are tabulated per (k, z_k) and
    gathered; the SLO slack of every class is then one product with pi.  Returns (z, its
    objective); the current z when nothing is feasible."""
    a = pi.sum(axis=1)
    load = (p.arrival[:, None] * pi * T).sum(axis=0)           # U_k
    rate = (p.arrival[:, None] * pi).sum(axis=0)
    routed = rate > 0
    tbar = np.where(routed, load / np.where(routed, rate, 1.0), 0.0)
    u_ik = p.arrival[:, None] * T
    r_t = _reservation(p, eta)[:, None] - delta * p.L_pre[:, None]
    capload = (1.0 + p.kappa) * (u_ik * pi * r_t).sum(axis=0)   # z_k times the capacity term
    prefix = (delta * p.L_pre[:, None]).sum(axis=0)
    zmax = int(Z.max()) if Z.size else 0
    ok_t = np.zeros((p.nK, zmax + 1), bool)
    W_t = np.zeros((p.nK, zmax + 1))
    for k in range(p.nK):
        ok_t[k, 0] = not routed[k]
        for v in range(1, zmax + 1):
            u = load[k] / v
            ok = u <= p.u_max * (1 + 1e-9) and u < 1.0
            ok = ok and capload[k] / v + prefix[k] - p.M[k] <= 1e-7 * max(p.M[k], 1.0)
            ok_t[k, v] = ok
            if ok and routed[k]:
                W_t[k, v] = u * (1.0 + cv2[k]) / (2.0 * (1.0 - u)) * tbar[k]
    base = (pi * T).sum(axis=1) - a * p.D                     # [I]
    wslo = p.arrival * p.c_slo
    gpu = (pi * p.c_gpu * (p.tau * p.pp)[None, :] * T).sum(axis=1)
    const = float((p.arrival * (a * d + gpu + (1.0 - a) * p.c_rej)).sum())
    kk = np.arange(p.nK)[None, :]
    vals_all = np.empty(Z.shape[0])
    for s0 in range(0, Z.shape[0], chunk):
        zc = Z[s0:s0 + chunk]
        ok = np.all(ok_t[kk, zc], axis=1)
        lat = W_t[kk, zc] @ pi.T + base[None, :]               # [n, I]
        val = const + np.maximum(lat, 0.0) @ wslo
        val[~ok] = np.inf
        vals_all[s0:s0 + chunk] = val
    best_idx = int(np.argmin(vals_all))
    best_val = float(vals_all[best_idx])
    cur = np.flatnonzero(np.all(Z == z_cur[None, :], axis=1))
    if cur.size and np.isfinite(vals_all[cur[0]]) and vals_all[cur[0]] <= best_val * (1 + 1e-12) + 1e-12:
        return z_cur.copy(), float(vals_all[cur[0]])
    if not np.isfinite(best_val):
        return z_cur.copy(), np.inf
    return Z[best_idx].copy(), best_val


# ---------------------------------------------------------------- Alg. 1

def initial_z(p: Problem) -> np.ndarray:
    """z^(0): one group of each configuration in ascending order of GPUs per group (ties by
    index), round after round, while the budget allows -- every configuration that fits is
    deployed, so LP1 can route to any of them from the start."""
    g = (p.tau * p.pp).astype(np.int64)
    order = sorted(range(p.nK), key=lambda k: (int(g[k]), k))
    z = np.zeros(p.nK, np.int32)
    left = int(p.J)
    while True:
        placed = False
        for k in order:
            if g[k] <= left and p.M[k] > 0:
                z[k] += 1
                left -= int(g[k])
                placed = True
        if not placed:
            return z


def solve(p: Problem, tables: Tables, T_max: int = 20, inner_max: int = 100, steps: int = 7,
          tol: float = 1e-9, Z: Optional[np.ndarray] = None, z0: Optional[np.ndarray] = None,
          log=None) -> BcdResult:
    """Alg. 1: Block 1 (LP1 / LP2 alternation), Block 2, Block 3, until (z, delta) repeats.

    LP1 holds the waiting times at those of the current routing; its solution pi' is taken
    along the segment from the current pi (step 1, 1/2, ..., 2^(1 - steps); LP1's feasible
    set is convex, so every point of it is feasible) at the first step that lowers the
    objective of eq. dro_obj, then LP2 re-optimises r exactly.  Block 1 ends when a round
    lowers the objective by less than ``tol`` (relative) or after ``inner_max`` rounds.
    Block 3 keeps z unless another z is strictly better, so no block update raises the
    objective (the premise of Prop. "Convergence").  ``z0`` replaces the default first
    deployment (a warm start from the deployment in service)."""
    t_all = time.perf_counter()
    secs = {"tables": tables.seconds, "lp1": 0.0, "lp2": 0.0, "block2": 0.0, "block3": 0.0}
    T = service_time(p)
    cv2 = service_cv2(p)
    t0 = time.perf_counter()
    if Z is None:
        Z = config_set(p.tau * p.pp, p.J)
    secs["enumerate_Z"] = time.perf_counter() - t0
    z = initial_z(p) if z0 is None else np.asarray(z0, np.int32).copy()
    if int((z * p.tau * p.pp).sum()) > p.J or np.any(z < 0):
        raise ValueError("z0 is outside the configuration set")
    delta = np.zeros((p.I, p.nK), np.int32)
    eta = tables.eta0.astype(np.int64).copy()
    d = tables.d0.copy()              # gamma^(0) eps + S(eta^(0), gamma^(0)) until the first LP2
    pi = np.zeros((p.I, p.nK))
    history: List[dict] = []
    trace: List[float] = []
    lp_rounds = 0
    t = 0
    cur = objective(p, T, cv2, tables, z, eta, pi, delta, d=d)[0]
    trace.append(cur)
    for t in range(1, T_max + 1):
        for _ in range(inner_max):
            W = waiting_time(p, T, cv2, pi, z)
            t0 = time.perf_counter()
            prop = lp1(p, T, W, z, eta, delta, d)
            secs["lp1"] += time.perf_counter() - t0
            lp_rounds += 1
            start = cur
            step = 1.0
            for _ in range(steps):
                cand = pi + step * (prop - pi)
                val = objective(p, T, cv2, tables, z, eta, cand, delta, d=d)[0]
                if val < cur:
                    pi, cur = cand, val
                    break
                step *= 0.5
            t0 = time.perf_counter()
            eta_new = lp2(p, T, tables, z, pi, delta, eta)
            secs["lp2"] += time.perf_counter() - t0
            d_new = tables.cost[np.arange(p.I), eta_new]
            val = objective(p, T, cv2, tables, z, eta_new, pi, delta, d=d_new)[0]
            if val <= cur:
                eta, d, cur = eta_new, d_new, val
            trace.append(cur)
            if not (cur < start - tol * max(abs(start), 1.0)):
                break
        t0 = time.perf_counter()
        delta_new = block2(p, T, z, pi)
        secs["block2"] += time.perf_counter() - t0
        val = objective(p, T, cv2, tables, z, eta, pi, delta_new, d=d)[0]
        if val <= cur:                # the rule as printed never helps feasibility less than this
            cur = val
        else:
            delta_new = delta
        trace.append(cur)
        t0 = time.perf_counter()
        z_new, val = block3(p, T, cv2, Z, z, eta, pi, delta_new, d)
        secs["block3"] += time.perf_counter() - t0
        if val <= cur:
            cur = val
        else:
            z_new = z
        trace.append(cur)
        history.append({"t": t, "z": z_new.tolist(), "delta_ones": int(delta_new.sum()), "objective": cur,
                        "lp_rounds": lp_rounds})
        if log:
            log(f"BCD iteration {t}: z={z_new.tolist()} objective={cur:.9g} lp_rounds={lp_rounds}")
        same = np.array_equal(z_new, z) and np.array_equal(delta_new, delta)
        z, delta = z_new, delta_new
        if same:
            break
    total, parts, s, W = objective(p, T, cv2, tables, z, eta, pi, delta, d=d)
    secs["total"] = time.perf_counter() - t_all + tables.seconds
    res = BcdResult(z=z, r=p.L_in.astype(np.int64) + eta, eta=eta, gamma=tables.gamma[np.arange(p.I), eta], pi=pi,
                    delta=delta, s=s, W=W, objective=float(total), parts=parts, outer_iterations=t,
                    lp_rounds=lp_rounds, history=history, seconds=secs)
    res.trace = trace
    return res


# ---------------------------------------------------------------- the library's part

def gpu_tables(p: Problem, device: int = 0) -> Tables:
    """f_i(eta) for every integer eta in [0, L_max^i] (one ``kvdro_eval_dual`` per distinct
    L_max, all classes of that support size at once; class i takes radius eps_i) and the
    initial cost gamma^(0) eps_i + S_i(eta0_i, gamma^(0)) with gamma^(0) = c_p
    (``kvdro_eval_grid`` in ENVELOPE mode)."""
    from . import kvdro as kv

    t0 = time.perf_counter()
    I = p.I
    Lmax = int(p.L_max.max())
    cost = np.full((I, Lmax + 1), np.inf)
    gamma = np.full((I, Lmax + 1), np.nan)
    eta0 = np.clip(np.rint(p.mean_output()), 0, p.L_max).astype(np.int64)
    d0 = np.empty(I)
    for L in np.unique(p.L_max):
        idx = np.flatnonzero(p.L_max == L)
        n = idx.size
        parts = [p.class_samples(i) for i in idx]
        off = np.zeros(n + 1, np.int64)
        off[1:] = np.cumsum([x.size for x in parts])
        smp = np.ascontiguousarray(np.concatenate(parts), np.int32)
        ctx = kv.kvdro_create(device)
        try:
            kv.kvdro_load_samples(ctx, n, off, smp, np.full(n, L, np.int32), np.zeros(n, np.int32))
            R = int(L) + 1
            grid = np.arange(R, dtype=np.int32)
            eps = np.ascontiguousarray(p.eps[idx], np.float64)
            c = np.empty((1, n, n, R), np.float64)
            g = np.empty((1, n, n, R), np.float64)
            kv.kvdro_eval_dual(ctx, R, grid, n, eps, 1, [p.c_p], [p.c_w], cost=c, gamma=g)
            e0 = np.unique(eta0[idx]).astype(np.int32)
            c0 = np.empty((1, n, n, e0.size), np.float64)
            kv.kvdro_eval_grid(ctx, kv.KVDRO_ENVELOPE, e0.size, e0, 1, [p.c_p], n, eps, 1, [p.c_p], [p.c_w], cost=c0)
        finally:
            kv.kvdro_destroy(ctx)
        for j, i in enumerate(idx):
            cost[i, :R] = c[0, j, j]
            gamma[i, :R] = g[0, j, j]
            d0[i] = c0[0, j, j, int(np.searchsorted(e0, eta0[i]))]
    return Tables(cost=cost, gamma=gamma, eta0=eta0, d0=d0, seconds=time.perf_counter() - t0)


def main():
    import argparse
    import os
    import sys

    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    from synth import bcd_instance

    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--classes", type=int, default=5)
    ap.add_argument("--configs", type=int, default=4)
    ap.add_argument("--samples", type=int, default=1000)
    ap.add_argument("--gpus", type=int, default=8, help="GPU budget J of the modelled cluster")
    ap.add_argument("--rho", type=float, default=10.0)
    ap.add_argument("--load", type=float, default=0.6)
    ap.add_argument("--device", type=int, default=0)
    a = ap.parse_args()
    p = Problem(**bcd_instance(a.classes, a.configs, a.samples, a.gpus, rho=a.rho, load=a.load))
    res = solve(p, gpu_tables(p, a.device), log=lambda s: print(s, file=sys.stderr))
    print(json.dumps(res.to_json()))


if __name__ == "__main__":
    main()
