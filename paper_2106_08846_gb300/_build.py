"""In-tree build of the CUDA library (libbsr_gb300.so) for sm_103a with nvcc.

Translation units compile in parallel into ``_build/`` beside this file and
link into ``libbsr_gb300.so``; nothing is installed. A unit is recompiled when
it or any header it may include is newer than its object file.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
from typing import List

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OBJDIR = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libbsr_gb300.so")
PROBE_SRC = os.path.join(PKG, "probe", "fp32_peak.cu")
PROBE_LIB = os.path.join(PKG, "libbsr_probe.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
         "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build libbsr_gb300.so")


def sources() -> List[str]:
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")) + glob.glob(os.path.join(CSRC, "*.cpp")))


def _headers() -> List[str]:
    return glob.glob(os.path.join(CSRC, "*.h")) + glob.glob(os.path.join(CSRC, "*.cuh")) + \
        glob.glob(os.path.join(INCLUDE, "*.h"))


def _stale(target: str, deps: List[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _compile(src: str, extra: List[str]) -> str:
    obj = os.path.join(OBJDIR, os.path.basename(src) + ".o")
    if _stale(obj, [src] + _headers()):
        tmp = obj + f".{os.getpid()}.tmp"
        cmd = [nvcc()] + ARCH + FLAGS + extra + ["-c", src, "-o", tmp]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, obj)
    return obj


def build_probe(force: bool = False) -> str:
    """The benchmark's FP32 FMA peak probe (libbsr_probe.so, not part of the C ABI)."""
    if force or _stale(PROBE_LIB, [PROBE_SRC]):
        tmp = PROBE_LIB + f".{os.getpid()}.tmp"
        cmd = [nvcc()] + ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-shared", PROBE_SRC,
                                 "-o", tmp, "-lcudart_static"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {PROBE_SRC}:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, PROBE_LIB)
    return PROBE_LIB


def build(force: bool = False, extra: List[str] = (), jobs: int = 0) -> str:
    """Compile every unit under csrc/ and link libbsr_gb300.so (and the peak
    probe, libbsr_probe.so); returns the library's path."""
    os.makedirs(OBJDIR, exist_ok=True)
    if force:
        for o in glob.glob(os.path.join(OBJDIR, "*.o")):
            os.remove(o)
    srcs = sources()
    with cf.ThreadPoolExecutor(max_workers=jobs or min(len(srcs) + 1, os.cpu_count() or 4)) as ex:
        probe = ex.submit(build_probe, force)
        objs = list(ex.map(lambda s: _compile(s, list(extra)), srcs))
        probe.result()
    if _stale(LIB, objs):
        tmp = LIB + f".{os.getpid()}.tmp"
        cmd = [nvcc()] + ARCH + ["-shared", "-o", tmp] + objs + ["-lcudart_static"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build())
