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
