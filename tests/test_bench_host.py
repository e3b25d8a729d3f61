"""Host logic of bench.py: multi-rank aggregation (gloo, world size 2, CPU), the clock
parser, the reference arm's rank handling and the ncu-summary staleness check."""

import json
import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

torch = pytest.importorskip("torch")


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        slowest = bench.reduce_max(1.0 + rank)            # rank 1 is the slow one
        q.put((rank, slowest, bench.weak_scaling_value(100, 10, world, slowest)))
    finally:
        dist.destroy_process_group()


def test_multi_rank_max_and_weak_value():
    import socket
    import torch.multiprocessing as mp
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [2.0, 2.0]
    assert all(r[2] == 100 * 10 * 2 / 2.0 for r in res)


def test_single_process_reduce_is_identity():
    assert bench.reduce_max(3.5) == 3.5


def test_clock_sampler_parses_nvidia_smi_rows(tmp_path):
    cs = bench.ClockSampler("0")
    cs.path = str(tmp_path / "c.csv")
    open(cs.path, "w").write(
        "0, 1965, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n"
        "0, 1980, 2070, 950.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n"
        "0, 1995, 2070, 990.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n")

    class Done:
        def terminate(self):
            pass

        def wait(self, timeout=None):
            return 0

    cs.proc = Done()
    cs.fh = open(os.devnull, "w")
    out = cs.stop()
    assert out["sm_mhz"] == 1980 and out["sm_max_mhz"] == 2070 and out["reasons"] == ["sw_power_cap"]


def test_reference_arm_only_rank0_prints():
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_reference_arm_line_has_the_contract_keys():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr
    line = json.loads(r.stdout.strip().splitlines()[-1])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["value"] > 0


def test_stale_profile_is_not_reported(tmp_path, monkeypatch):
    prof = tmp_path / "p.md"
    prof.write_text("grid_cu_sha256: " + "0" * 64 + "\ntraffic_bytes_per_launch: 123\ninst_per_term: 1.1\n")
    monkeypatch.setattr(bench, "PROFILE", str(prof))
    assert bench.profile_figures() == (None, None)
    import hashlib
    h = hashlib.sha256(open(bench.GRID_SOURCE, "rb").read()).hexdigest()
    prof.write_text(f"grid_cu_sha256: {h}\ntraffic_bytes_per_launch: 123\ninst_per_term: 1.1\n")
    assert bench.profile_figures() == (123.0, 1.1)


def test_oracle_sample_rows_stride_over_regimes_and_reservations():
    """The CPU-baseline sample: strided (regime, r) rows, each with every class and lam value."""
    from synth import regime_sweep_workload_k8_n2e5
    w = regime_sweep_workload_k8_n2e5()
    (m, k, r, l), terms = bench.oracle_rows(w, 4)
    M, K, R, NL = len(w.cp), w.K, len(w.r), len(w.lam)
    assert m.size == 4 * K * NL and terms == 4 * NL * int(w.N.sum())
    assert m[0] == 0 and r[0] == 0 and m[-1] == M - 1 and r[-1] == R - 1
    assert set(np.unique(k)) == set(range(K)) and set(np.unique(l)) == set(range(NL))


def test_case_spec_options():
    w, mode = bench.case_workload("regimes_k8_n2e5:fp32:m=16,nl=256,L=4194305,rstride=4")
    assert mode == "fp32" and len(w.cp) == 16 and len(w.lam) == 256 and len(w.r) == 512
    assert (w.L == 4194305).all() and w.lam[0] == 1e-3 and abs(w.lam[-1] - 1e3) < 1e-9
    assert bench.case_options("regimes_k8_n2e5:fp32:m=16,out=all") == {"m": "16", "out": "all"}
    assert bench.case_options("regimes_k8_n2e5:fp32") == {}
