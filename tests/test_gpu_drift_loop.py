"""The drifting-workload loop: per-iteration records, resume, and agreement with a direct grid pass."""

import json

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2607_16892_gb300 import kvdro  # noqa: E402
from paper_2607_16892_gb300.drift_loop import run as drift_run  # noqa: E402
from paper_2607_16892_gb300.runner import run  # noqa: E402
from synth import drift_loop_workload_k32_n1e6  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_drift_loop_records_resume_and_match_a_direct_pass(tmp_path):
    out = str(tmp_path / "drift.jsonl")
    first = drift_run(iterations=2, out=out, log=lambda *_: None)
    assert [r["iteration"] for r in first] == [0, 1]
    again = drift_run(iterations=3, out=out, resume=True, log=lambda *_: None)
    assert [r["iteration"] for r in again] == [2]
    lines = [json.loads(l) for l in open(out)]
    assert [l["iteration"] for l in lines] == [0, 1, 2]
    for rec in lines:
        assert rec["gpu_ms"] >= rec["eval_ms"] > 0 and rec["terms_per_s"] > 0
        assert all(0.0 <= f <= 1.0 for f in rec["fhat_eps0"])
    # iteration 1 chose the same reservations as a direct pass over the same workload
    w = drift_loop_workload_k32_n1e6(1)
    direct = run(w, kvdro.KVDRO_FP32, outputs=("r_idx",))
    assert lines[1]["r_star_eps0"] == w.r[direct["r_idx"][0, 0]].tolist()
    # medians drift upward with the +2 % per iteration medians
    assert np.mean(lines[2]["median_quantile"]) > np.mean(lines[0]["median_quantile"])
