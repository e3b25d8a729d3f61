"""Seeded instances of the joint configuration / routing / caching / reservation problem.

The paper's evaluation (Sec. 5.1 "System Configuration") models J = 8 A100-80GB GPUs
serving a 70B model with configurations (TP, PP) in {(2,1), (4,1), (2,2), (4,2)} and the
weights c_p/c_w = 10, c_slo/c_w = 5, c_rej/c_w = 5000, kappa = 0.2; its scalability table
(Sec. 5.2) grows the instance to 15 classes, 12 configurations, N = 2000 samples and a
48-GPU cluster.  It does not print the serving-model constants (alpha, beta, C_k, B_k,
M_k, t_ar, c_gpu), the classes' input lengths, prefixes, SLOs or arrival rates, nor the
extra configurations; the values below stand in for them and are stated here:

  * KV capacity of a group: (76 GB x tau p - 140 GB of FP16 weights) / 327,680 bytes per
    token (80 layers x 8 KV heads x 128 dims x K and V x 2 bytes);
  * effective compute C_k = tau p x 156 TFLOP/s (half of the A100's 312 dense FP16),
    effective decode bandwidth B_k = tau x 1.43 TB/s (70% of 2.04 TB/s; a sequence's decode
    crosses the pipeline stages one after another, so PP adds no bandwidth);
  * alpha = 1.4e11 FLOP per prefill token, beta = 1.4e11 bytes per decode token,
    N_L = 80, t_ar = 10 us, c_gpu = 1 per GPU-second;
  * class archetypes (input length, shared prefix, median output, sigma, SLO) cycle over
    chat, code, summarisation, QA, reasoning and long-document; output lengths are
    lognormal, rounded and clipped to [1, L_max];
  * arrival rates: every class offers the same load, scaled so that all classes on
    J / 4 TP4 groups would run at ``load`` x u_max utilisation;
  * eps_i = 0.15 E[xi_i] (Sec. 5.1 "Default knobs").

Seeds: numpy PCG64(20260000 + 60000 + 1000 * variant + class).
"""

from __future__ import annotations

from typing import Dict

import numpy as np

# name, input length, shared prefix, median output, sigma, SLO (s), L_max
_ARCHETYPES = (
    ("chat", 400, 200, 150.0, 0.9, 20.0, 8192),
    ("code", 2000, 1500, 60.0, 1.0, 8.0, 8192),
    ("summarise", 6000, 500, 300.0, 0.6, 30.0, 8192),
    ("qa", 150, 100, 40.0, 0.8, 6.0, 8192),
    ("reasoning", 800, 300, 1500.0, 0.7, 120.0, 32768),
    ("long_document", 28000, 4000, 1200.0, 0.9, 90.0, 32768),
)

# (TP, PP): the paper's four first, then further candidates for the larger instances
CONFIGS = ((2, 1), (4, 1), (2, 2), (4, 2), (8, 1), (2, 4), (8, 2), (4, 4), (1, 2), (1, 4), (8, 4), (16, 1))

# the scalability instances (classes, configurations, samples per class, GPU budget)
SCALABILITY_SIZES = ((3, 4, 100, 8), (4, 4, 150, 8), (5, 5, 200, 16), (6, 6, 300, 16), (8, 6, 500, 16),
                     (10, 8, 1000, 32), (15, 12, 2000, 48))

_GB = 1e9
_KV_BYTES_PER_TOKEN = 80 * 8 * 128 * 2 * 2


def bcd_instance(n_classes: int, n_configs: int, n_samples: int, J: int, rho: float = 10.0, load: float = 0.6,
                 variant: int = 0, u_max: float = 0.95, L_cap: int = 0) -> Dict:
    """Keyword arguments of ``paper_2607_16892_gb300.bcd.Problem`` for one seeded instance.
    ``L_cap`` > 0 caps every class's maximum output length (small cases for CPU tests)."""
    if not 1 <= n_configs <= len(CONFIGS):
        raise ValueError(f"n_configs must be in [1, {len(CONFIGS)}]")
    tau = np.array([CONFIGS[k][0] for k in range(n_configs)], np.int64)
    pp = np.array([CONFIGS[k][1] for k in range(n_configs)], np.int64)
    g = tau * pp
    M = np.floor((76 * _GB * g - 140 * _GB) / _KV_BYTES_PER_TOKEN)
    M = np.maximum(M, 0.0)
    C = g * 156e12
    B = tau * 1.43e12
    alpha, beta, n_layers, t_ar = 1.4e11, 1.4e11, 80, 1e-5

    L_in, L_pre, D, L_max, cls = [], [], [], [], []
    for i in range(n_classes):
        name, lin, lpre, med, sig, slo, lmax = _ARCHETYPES[i % len(_ARCHETYPES)]
        if L_cap > 0:
            lmax = min(lmax, int(L_cap))
        rng = np.random.Generator(np.random.PCG64(20260000 + 60000 + 1000 * variant + i))
        scale = float(rng.uniform(0.8, 1.25))
        L_in.append(int(round(lin * scale)))
        L_pre.append(min(int(round(lpre * scale)), L_in[-1]))
        D.append(slo)
        L_max.append(lmax)
        x = np.rint(np.exp(np.log(med * float(rng.uniform(0.8, 1.25))) + sig * rng.standard_normal(n_samples)))
        cls.append(np.clip(x, 1, lmax).astype(np.int32))
    offsets = np.zeros(n_classes + 1, np.int64)
    offsets[1:] = np.cumsum([c.size for c in cls])
    samples = np.concatenate(cls).astype(np.int32)
    L_in = np.array(L_in, np.int64)
    mean = np.array([c.mean() for c in cls])
    # reference service time on a TP4 group: alpha L_in / (4 x 156e12) + beta E[xi] / (4 x 1.43e12)
    t_ref = alpha * L_in / (4 * 156e12) + beta * mean / (4 * 1.43e12) + n_layers * 4 * t_ar
    arrival = load * u_max * (J / 4.0) / (n_classes * t_ref)
    return dict(arrival=arrival, L_in=L_in, L_pre=np.array(L_pre, np.int64), D=np.array(D, np.float64),
                L_max=np.array(L_max, np.int64), samples=samples, offsets=offsets, eps=0.15 * mean,
                J=int(J), tau=tau, pp=pp, M=M, C=C.astype(np.float64), B=B.astype(np.float64), alpha=alpha,
                beta=beta, n_layers=n_layers, t_ar=t_ar, c_p=float(rho), c_w=1.0, c_gpu=1.0, c_slo=5.0,
                c_rej=5000.0, kappa=0.2, u_max=u_max,
                name=f"bcd_i{n_classes}_k{n_configs}_n{n_samples}_j{J}_rho{rho:g}")
