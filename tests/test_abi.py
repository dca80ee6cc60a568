"""The C ABI library: it builds, loads and exports every function include/bsr.h
declares; argument checks that return before any device work behave as
documented. No compute call runs here (no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bsr.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2106_08846_gb300 import _build
    _build.build()
    import paper_2106_08846_gb300 as pkg
    return pkg.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(bsr_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("bsr_from_dense", "bsr_create", "bsr_reserve", "bsr_spmm", "bsr_check_device_status",
              "bsr_get_schedule", "bsr_destroy", "bsr_status_str"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2106_08846_gb300 import bsrlib
    out = subprocess.run(["nm", "-D", "--defined-only", bsrlib.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (bsr_\w+)$", out, flags=re.M))
    for n in declared_functions():
        assert n in exported, n
        assert hasattr(lib, n)


def test_header_compiles_as_c():
    src = '#include "bsr.h"\nint main(void){ return (int)BSR_OK + (int)BSR_F32; }\n'
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                        "-x", "c", "-fsyntax-only", "-"], input=src, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_status_codes_match_header(lib):
    from paper_2106_08846_gb300 import bsrlib
    src = open(HEADER).read()
    for name, val in re.findall(r"\b(BSR_(?:OK|ERR_\w+))\s*=\s*(\d+)", src):
        assert getattr(bsrlib, name) == int(val)
        assert lib.bsr_status_str(int(val)).decode() == name
    assert lib.bsr_status_str(999).decode() == "BSR_ERR_UNKNOWN"


def test_host_side_argument_errors(lib):
    from paper_2106_08846_gb300 import bsrlib as b
    P = ctypes.c_void_p
    out = P()
    # shape and argument checks run before any CUDA call
    assert lib.bsr_create(None, None, None, 32, 1, 768, 768, 0, None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_create(None, None, None, 32, 1, 770, 768, 0, ctypes.byref(out)) == b.BSR_ERR_SHAPE
    assert lib.bsr_create(None, None, None, 0, 1, 768, 768, 0, ctypes.byref(out)) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_create(None, None, None, 128, 64, 768, 768, 0, ctypes.byref(out)) == b.BSR_ERR_UNSUPPORTED
    assert lib.bsr_create(None, None, None, 32, 1, 768, 768, 7, ctypes.byref(out)) == b.BSR_ERR_UNSUPPORTED
    assert lib.bsr_create(None, None, None, 32, 1, 768, 768, 0, ctypes.byref(out)) == b.BSR_ERR_INVALID_ARG
    n = ctypes.c_int64(0)
    assert lib.bsr_from_dense(None, 768, 770, 32, 4, 0.0, 0, None, None, None, 0, ctypes.byref(n),
                              None) == b.BSR_ERR_SHAPE
    dummy = ctypes.c_void_p(16)
    assert lib.bsr_from_dense(dummy, 64, 64, 8, 8, -1.0, 0, dummy, None, None, 0, ctypes.byref(n),
                              None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_from_dense(dummy, 64, 64, 8, 8, float("nan"), 0, dummy, None, None, 0,
                              ctypes.byref(n), None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_from_dense(dummy, 64, 64, 8, 8, 0.0, 0, None, None, None, 0, ctypes.byref(n),
                              None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_from_dense(dummy, 64, 64, 8, 8, 0.0, 0, dummy, None, None, 5, ctypes.byref(n),
                              None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_spmm(None, None, None, None, 4, None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_reserve(None, 4) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_check_device_status(None) == b.BSR_ERR_INVALID_ARG
    buf = ctypes.create_string_buffer(16)
    assert lib.bsr_get_schedule(None, buf, 16) == b.BSR_ERR_INVALID_ARG
    lib.bsr_destroy(None)
    # plans: argument checks before any CUDA call
    plan = P()
    assert lib.bsr_plan_create(None, None, None, None, None, 0, 0, None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_plan_create(None, None, None, None, None, -1, 0, ctypes.byref(plan)) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_plan_create(None, None, None, None, None, 2, 1, ctypes.byref(plan)) == b.BSR_ERR_INVALID_ARG
    assert plan.value is None
    assert lib.bsr_plan_launch(None, None) == b.BSR_ERR_INVALID_ARG
    assert lib.bsr_plan_get_order(None, None, None, 0, None) == b.BSR_ERR_INVALID_ARG
    lib.bsr_plan_destroy(None)


def test_parse_schedule():
    from paper_2106_08846_gb300.bsrlib import parse_schedule
    d = parse_schedule("variant=xstage\nitems=24\nsplit_len=0\n")
    assert d == {"variant": "xstage", "items": 24, "split_len": 0}


def test_product_path_has_no_cpu_fallback():
    """The package never imports the oracle; nothing under it computes on the host."""
    pkg = os.path.join(ROOT, "paper_2106_08846_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cpp", ".cu", ".h", ".cuh")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "ref_bsr" not in text, f
