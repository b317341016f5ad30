"""The C ABI library loads and exports every entry point include/pkv.h declares."""
import os
import re

from paper_2605_11232_gb300 import pkv

from _lib import built_lib

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared(header):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(\w+)\s*\(", text, flags=re.M)))


def test_every_declared_symbol_is_exported():
    lib = built_lib()
    names = _declared("pkv.h")
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(pkv.EXPORTS)


def test_last_error_is_a_string():
    built_lib()
    assert isinstance(pkv.pkv_last_error(), str)


def test_header_is_plain_c_and_host_calls_work_from_c(tmp_path):
    """include/pkv.h compiles as C11 (-Wall -Wextra -Werror), and a plain C
    program linked against libpkv.so drives the host-side calls: pool, prefix
    cache, slot mapping, prefix groups (tests/c/host_abi.c)."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        import pytest
        pytest.skip("no gcc")
    lib = pkv.LIB_PATH
    built_lib()
    exe = str(tmp_path / "host_abi")
    subprocess.check_call(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-I",
                           os.path.join(ROOT, "include"), os.path.join(ROOT, "tests", "c", "host_abi.c"),
                           "-o", exe, "-L", os.path.dirname(lib), "-lpkv",
                           "-Wl,-rpath," + os.path.dirname(lib)])
    out = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == "ok"
