"""The C ABI from a plain C program: tests/c_consumer/kvdro_consumer.c includes only kvdro.h,
passes host buffers only (no CUDA header, no device memory of its own) and prints what the
library returns.  On any machine it must compile with -Werror and link against libkvdro.so; on
a GPU its outputs must match the oracle."""

import os
import subprocess

import numpy as np
import pytest

from paper_2607_16892_gb300 import build as kbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c_consumer", "kvdro_consumer.c")


def build_consumer(tmp_path) -> str:
    lib = kbuild.build()
    libdir = os.path.dirname(lib)
    exe = str(tmp_path / "kvdro_consumer")
    subprocess.run(["gcc", "-std=c99", "-O2", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"), SRC,
                    "-L", libdir, "-lkvdro", f"-Wl,-rpath,{libdir}", "-o", exe], check=True)
    return exe


def test_a_plain_c_program_compiles_and_links_against_the_library(tmp_path):
    exe = build_consumer(tmp_path)
    assert os.access(exe, os.X_OK)
    out = subprocess.run(["ldd", exe], capture_output=True, text=True).stdout
    assert "libkvdro.so" in out and "not found" not in out


def _input_text(w, precision: int) -> str:
    parts = [str(w.K), " ".join(map(str, w.offsets)), " ".join(map(str, w.samples)), " ".join(map(str, w.L)),
             " ".join(map(str, w.L_in)), str(len(w.r)), " ".join(map(str, w.r)), str(len(w.lam)),
             " ".join(repr(float(v)) for v in w.lam), str(len(w.eps)), " ".join(repr(float(v)) for v in w.eps),
             str(len(w.cp)), " ".join(repr(float(v)) for v in w.cp), " ".join(repr(float(v)) for v in w.cw),
             str(len(w.fractiles)), " ".join(repr(float(v)) for v in w.fractiles), str(precision)]
    return "\n".join(parts) + "\n"


def _parse(text: str, w) -> dict:
    M, E, K, R = len(w.cp), len(w.eps), w.K, len(w.r)
    shapes = {"quant": (K, len(w.fractiles)), "sorted": (int(w.offsets[-1]),), "cost": (M, E, K, R),
              "lam_idx": (M, E, K, R), "r_idx": (M, E, K), "min_cost": (M, E, K), "fhat": (M, E, K)}
    out = {}
    for line in text.splitlines():
        name, n, *vals = line.split()
        assert name in shapes, line[:200]
        dt = np.float64 if name in ("cost", "min_cost", "fhat") else np.int32
        a = np.array([float(v) for v in vals] if dt == np.float64 else [int(v) for v in vals], dt)
        assert a.size == int(n) == int(np.prod(shapes[name])), name
        out[name] = a.reshape(shapes[name])
    assert set(out) == set(shapes)
    return out


@pytest.mark.gpu
@pytest.mark.parametrize("mode", ["exact", "fp64", "envelope"])
def test_the_c_programs_outputs_match_the_oracle(tmp_path, mode):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from oracle import oracle as O
    from paper_2607_16892_gb300 import kvdro
    from synth import random_case
    from tests.parity import compare_full

    exe = build_consumer(tmp_path)
    w = random_case(77, K=3, N=(4100, 515, 37), L=(2500, 2500, 2500), L_in=(0, 10, 3), R=41, n_lam=33, n_eps=3,
                    M=2, lam_range=(1e-3, 100.0), eps_max=200.0)
    prec = {"exact": kvdro.KVDRO_EXACT, "fp64": kvdro.KVDRO_FP64, "envelope": kvdro.KVDRO_ENVELOPE}[mode]
    res = subprocess.run([exe], input=_input_text(w, prec), capture_output=True, text=True, timeout=300)
    assert res.returncode == 0, res.stdout[-2000:] + res.stderr[-2000:]
    got = _parse(res.stdout, w)
    compare_full(w, got, O.solve(w), "exact" if mode == "exact" else "fp64")
