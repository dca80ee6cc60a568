"""The C programs under tests/c: the oracle's self-checks in C (no GPU) and the
C ABI driven from plain C against the oracle (GPU). Each is compiled with gcc
here and must exit 0."""
import os
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CDIR = os.path.join(ROOT, "tests", "c")
ORACLE = os.path.join(ROOT, "oracle")
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _compile(tmp_path, name, extra):
    exe = os.path.join(str(tmp_path), name)
    cmd = ["gcc", "-std=c11", "-O2", "-Wall", "-Werror", "-ffp-contract=off", "-I", ORACLE,
           "-o", exe, os.path.join(CDIR, name + ".c"), os.path.join(ORACLE, "ref_bsr.c")] + extra + ["-lm"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe


def test_oracle_self_checks_in_c(tmp_path):
    exe = _compile(tmp_path, "test_oracle", [])
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "all checks passed" in r.stdout


@pytest.mark.gpu
def test_c_abi_from_c_matches_the_oracle(tmp_path):
    from paper_2106_08846_gb300 import _build
    lib = _build.build()
    libdir = os.path.dirname(lib)
    cudalib = os.path.join(CUDA, "lib64")
    exe = _compile(tmp_path, "test_capi", [
        "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"),
        "-L", libdir, "-lbsr_gb300", "-L", cudalib, "-lcudart",
        "-Wl,-rpath," + libdir, "-Wl,-rpath," + cudalib])
    r = subprocess.run([exe], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "all cases passed" in r.stdout
