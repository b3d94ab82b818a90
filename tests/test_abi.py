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


def _header_constants() -> dict:
    """Every `#define CASSPEC_X <int>` and every `CASSPEC_X = <int>` enumerator of the header."""
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    out = {}
    for name, val in re.findall(r"#define\s+CASSPEC_([A-Z0-9_]+)\s+(0x[0-9A-Fa-f]+|-?\d+)u?\b", src):
        out[name] = int(val, 0)
    for name, val in re.findall(r"\bCASSPEC_([A-Z0-9_]+)\s*=\s*(-?\d+)", src):
        out[name] = int(val)
    for name, expr in re.findall(r"#define\s+CASSPEC_([A-Z0-9_]+)\s+\((\d+)\s*\*\s*CASSPEC_MAX_TREE\)", src):
        out[name] = int(expr) * out["MAX_TREE"]
    return out


def test_binding_constants_match_the_header():
    """The binding's copies of the header's constants (status codes, capacities, skip flags, option
    bits, tensor ids, profiling kinds) are the header's values."""
    import paper_2510_26843_gb300 as cs

    h = _header_constants()
    pairs = {"MAX_TREE": "MAX_TREE", "TOPK_MAX": "TOPK_MAX", "DYTC_WORK": "DYTC_WORK", "DYTC_MAX_CLASS": "DYTC_MAX_CLASS", "SKIP_ATTN": "SKIP_ATTN",
             "SKIP_FFN": "SKIP_FFN", "OPT_PDL": "OPT_PDL", "OPT_GRAPHS": "OPT_GRAPHS", "OPT_TEST_STALL": "OPT_TEST_STALL", "OPT_W4_TC": "OPT_W4_TC",
             "OPT_W8_TC": "OPT_W8_TC", "OK": "OK"}
    for key in list(h):
        if key.startswith(("E_", "T_", "K_")):
            pairs[key] = key
    checked = 0
    for hname, pname in pairs.items():
        if hname in h and hasattr(cs, pname):
            assert getattr(cs, pname) == h[hname], (hname, getattr(cs, pname), h[hname])
            checked += 1
    assert checked >= 40, checked  # status codes, tensor ids and profiling kinds are all covered
