"""Baseline reservation rules priced by the exact dual, against the oracle and the paper's structure."""

import numpy as np
import pytest

from oracle import oracle as O
from synth import Workload, random_case

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import baselines  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_rules_and_costs_match_the_oracle():
    w = random_case(61, K=3, N=(2000, 300, 41), L=(1500, 1500, 1500), R=3, n_lam=2, n_eps=2, M=1)
    w.cp = np.array([2.0, 10.0, 100.0])
    w.cw = np.ones(3)
    eps = [5.0, 80.0]
    recs = baselines.compare(w, eps)
    quant = O.quantiles(w, [0.90, 0.95, 0.99])
    for rec in recs:
        m, k = rec["regime"], rec["class"]
        x = w.class_samples(k)
        assert rec["rules"]["p90"]["r"] == quant[k, 0]
        assert rec["rules"]["p95_block16"]["r"] == min(int(np.ceil(quant[k, 1] / 16) * 16), int(w.L[k]))
        assert rec["rules"]["p99"]["r"] == quant[k, 2]
        assert rec["rules"]["mean"]["r"] == int(np.ceil(x.mean()))
        assert rec["rules"]["lp_2sigma"]["r"] == min(int(np.ceil(x.mean() + 2 * x.std())), int(w.L[k]))
        # every priced rule against the oracle's exact dual at that reservation
        rs = sorted({v["r"] for v in rec["rules"].values()} | {d["r"] for d in rec["dro"]})
        one = Workload(name="b", samples=x.astype(np.int32), offsets=np.array([0, x.size]), L=w.L[k:k + 1].copy(),
                       L_in=w.L_in[k:k + 1].copy(), r=np.asarray(rs, np.int32), lam=np.array([1.0]),
                       eps=np.asarray(rec["eps"]), cp=w.cp[m:m + 1].copy(), cw=w.cw[m:m + 1].copy(),
                       fractiles=np.array([0.5]))
        ref = O.solve_dual(one)["cost"][0, :, 0, :]
        for v in list(rec["rules"].values()):
            i = rs.index(v["r"])
            np.testing.assert_allclose(v["cost"], ref[:, i], rtol=1e-9)
        for e, d in enumerate(rec["dro"]):
            # the DRO reservation is the best over every integer r, so no rule beats it
            assert all(d["cost"] <= v["cost"][e] * (1 + 1e-12) for v in rec["rules"].values())
            np.testing.assert_allclose(d["cost"], ref[e, rs.index(d["r"])], rtol=1e-9)
        # at radius 0 the SAA reservation is the critical-fractile quantile (Prop. 2)
        q = rec["critical_fractile"]
        assert rec["rules"]["saa"]["r"] == O.quantiles(one, [q])[0, 0]
