"""Resume bookkeeping of the drifting-workload loop (host only)."""

from paper_2607_16892_gb300.drift_loop import _done_iterations


def test_done_iterations_reads_completed_lines(tmp_path):
    p = tmp_path / "d.jsonl"
    p.write_text('{"iteration": 0, "gpu_ms": 1}\n{"iteration": 3}\nnot json\n{"other": 1}\n')
    assert _done_iterations(str(p)) == {0, 3}
    assert _done_iterations(str(tmp_path / "missing.jsonl")) == set()
