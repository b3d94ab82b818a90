"""The C-ABI library builds, loads without a GPU, and exports every entry point include/casspec.h
declares; the Python binding wraps each of them and nothing else.  No compute calls."""
from __future__ import annotations

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "casspec.h")


def _declared() -> list[str]:
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(casspec_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib_path():
    from paper_2510_26843_gb300 import build as b

    return b.build()


def test_header_declares_the_tree_step_api():
    names = _declared()
    for required in ("casspec_create_model", "casspec_tree_step", "casspec_accept_greedy", "casspec_kv_compact"):
        assert required in names


def test_library_exports_every_declared_symbol(lib_path):
    lib = ctypes.CDLL(lib_path)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_header(lib_path):
    import paper_2510_26843_gb300 as cs

    assert sorted(cs.EXPORTS) == _declared()
    lib = cs.load_library(lib_path)
    for n in cs.EXPORTS:
        assert getattr(lib, n).argtypes is not None


def test_only_casspec_symbols_are_exported(lib_path):
    out = os.popen(f"nm -D --defined-only {lib_path}").read()
    funcs = [l.split()[-1] for l in out.splitlines() if " T " in l]
    assert funcs and all(f.startswith("casspec_") for f in funcs), funcs[:10]


def test_status_strings_without_gpu(lib_path):
    import paper_2510_26843_gb300 as cs

    cs.load_library(lib_path)
    assert cs.status_string(cs.E_TREE) == "invalid tree or accepted path"
    assert cs.status_string(cs.OK) == "ok"
