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
