"""Host-side checks of the C ABI: the library builds for sm_103a, loads, and exports
every entry point include/kvdro.h declares.  No kernel is launched here."""

import ctypes
import os
import re
import subprocess

import pytest

from paper_2607_16892_gb300 import build as kbuild
from paper_2607_16892_gb300 import kvdro

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kvdro.h")


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:int|const char\s*\*)\s+(kvdro_\w+)\s*\(", text, re.M)))


def test_header_declares_the_binding_symbols():
    assert declared_symbols() == sorted(kvdro.SYMBOLS)


def test_library_builds_and_exports_every_declared_symbol():
    path = kbuild.build()
    lib = ctypes.CDLL(path)
    for name in declared_symbols():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT\s+(kvdro_\w+)$", out, re.M))
    assert set(declared_symbols()) <= exported


def test_header_is_plain_c(tmp_path):
    src = tmp_path / "use.c"
    src.write_text('#include "kvdro.h"\nint main(void) { kvdro_ctx* c = 0; return kvdro_destroy(c); }\n')
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), "-c", str(src),
                    "-o", str(tmp_path / "use.o")], check=True)


def test_null_context_calls_are_safe():
    lib = kvdro.load_library()
    assert lib.kvdro_destroy(None) == kvdro.KVDRO_OK
    assert lib.kvdro_last_error(None) == b"null context"
    assert lib.kvdro_sync(None) == kvdro.KVDRO_EINVAL
    assert lib.kvdro_load_samples(None, 1, None, None, None, None, None) == kvdro.KVDRO_EINVAL
    assert lib.kvdro_create(None, 0) == kvdro.KVDRO_EINVAL


def test_create_without_a_device_reports_an_error():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(kvdro.KvdroError):
        kvdro.kvdro_create(0)


def test_binding_rejects_mis_sized_arrays_before_calling_the_library(monkeypatch):
    """The binding checks every array length against the sizes the call is given (and outputs
    against the loaded context's class count) and raises ValueError without calling the library:
    a short buffer would otherwise be read or written past its end."""
    import numpy as np

    def no_library(*_a, **_k):
        raise AssertionError("the library was called")

    monkeypatch.setattr(kvdro, "load_library", no_library)
    off, L = np.array([0, 5, 9], np.int64), np.array([100, 100], np.int32)
    samples = np.arange(9, dtype=np.int32)
    with pytest.raises(ValueError, match="offsets"):
        kvdro.kvdro_load_samples(None, 3, off, samples, [100, 100, 100])
    with pytest.raises(ValueError, match="lengths"):
        kvdro.kvdro_load_samples(None, 2, off, samples[:8], L)
    with pytest.raises(ValueError, match="L_in"):
        kvdro.kvdro_load_samples(None, 2, off, samples, L, L_in=[0])
    grid = dict(R=3, r=[10, 20, 30], NL=2, lam=[0.5, 5.0], E=2, eps=[0.0, 1.0], M=1, c_p=[10.0], c_w=[1.0])
    for key, bad in (("r", [10, 20]), ("lam", [0.5]), ("eps", [0.0]), ("c_p", [1.0, 2.0]), ("c_w", [])):
        with pytest.raises(ValueError, match=key):
            kvdro.kvdro_eval_grid(None, kvdro.KVDRO_FP32, **{**grid, key: bad})
    # outputs against the class count of the samples the context holds (here: 2 classes)
    ctx = ctypes.c_void_p(0x1234)
    monkeypatch.setitem(kvdro._loaded, ctx.value, (2, 9))
    M, E, K, R, NL = 1, 2, 2, 3, 2
    for key, n in (("S", M * K * R * NL - 1), ("cost", M * E * K * R + 1), ("lam_idx", 1), ("r_idx", M * E * K - 1),
                   ("min_cost", 0), ("fhat", M * E * K + 2)):
        with pytest.raises(ValueError, match=key):
            kvdro.kvdro_eval_grid(ctx, kvdro.KVDRO_FP64, **grid, **{key: np.empty(n, np.float64 if key not in
                                                                                    ("lam_idx", "r_idx") else np.int32)})
    with pytest.raises(ValueError, match="out"):
        kvdro.kvdro_quantiles(ctx, 3, [0.1, 0.5, 0.9], np.empty(5, np.int32))
    with pytest.raises(ValueError, match="out"):
        kvdro.kvdro_sorted_samples(ctx, np.empty(8, np.int32))
    with pytest.raises(ValueError, match="cost"):
        kvdro.kvdro_eval_dual(ctx, 3, [10, 20, 30], 2, [0.0, 1.0], 1, [10.0], [1.0], cost=np.empty(11))
    # the allocation-free entry point: sizes, and outputs must be device memory
    na = dict(K=2, offsets=off, lengths=samples, L_max=L, L_in=None, **grid)
    with pytest.raises(ValueError, match="r_idx"):
        kvdro.kvdro_eval_grid_noalloc(**na, r_idx=np.empty(M * E * K - 1, np.int32))
    with pytest.raises(ValueError, match="CUDA tensor"):
        kvdro.kvdro_eval_grid_noalloc(**na, r_idx=np.empty(M * E * K, np.int32))
