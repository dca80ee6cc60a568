"""CPU oracle for the BSR product (Section 2.2) -- TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. The library it wraps (``ref_bsr.c``) is
plain C with double accumulation, written from the definitions; it shares no
code with the CUDA path.

Arrays cross as numpy: float32 for fp32 data, uint16 bit patterns for
bfloat16 data; int32 ``indptr``/``indices``; results come back as float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "libbsr_oracle.so")
_lib = None

F32, BF16 = 0, 1


def build(force: bool = False) -> str:
    """Compile ref_bsr.c into libbsr_oracle.so (gcc, no fused multiply-add)."""
    src = os.path.join(_HERE, "ref_bsr.c")
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "ref_bsr.h"))):
        tmp = _SO + f".{os.getpid()}.tmp"
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-o", tmp,
               src, "-lm"]
        try:   # OpenMP shares the float-accumulate baseline's block rows among cores
            subprocess.check_call(cmd[:1] + ["-fopenmp"] + cmd[1:], stderr=subprocess.DEVNULL)
        except subprocess.CalledProcessError:
            subprocess.check_call(cmd)
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_SO)
        P, I64, I = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        lib.ref_bsr_count.argtypes = [P, I, I64, I64, I, I, ctypes.c_float, P]
        lib.ref_bsr_count.restype = I64
        lib.ref_bsr_fill.argtypes = [P, I, I64, I64, I, I, ctypes.c_float, P, P, P]
        lib.ref_bsr_to_dense.argtypes = [I, I64, I64, I, I, P, P, P, P]
        for name in ("ref_bsr_spmm", "ref_bsr_err_bound"):
            getattr(lib, name).argtypes = [I, I64, I64, I, I, P, P, P, P, P, P, I64, P]
        lib.ref_dense_linear.argtypes = [I, I64, I64, P, P, P, P, I64, P]
        lib.ref_bsr_spmm_f32acc.argtypes = [I, I64, I64, I, I, P, P, P, P, P, P, I64, P, I]
        lib.ref_max_threads.restype = I
        lib.ref_round_f32.argtypes = [P, P, I64]
        lib.ref_round_bf16.argtypes = [P, P, I64]
        _lib = lib
    return _lib


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError(f"oracle takes float32 or uint16 (bf16 bits), not {a.dtype}")


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _rows(rows, N):
    if rows is None:
        return None, N
    r = np.ascontiguousarray(rows, dtype=np.int64)
    if r.size and (r.min() < 0 or r.max() >= N):
        raise IndexError("token index out of range")
    return r, r.size


def bsr_from_dense(W: np.ndarray, R: int, C: int, threshold: float = 0.0
                   ) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """(indptr, indices, data) of the dense W[M, K] in R x C blocks."""
    lib = _load()
    W = np.ascontiguousarray(W)
    dt = _dtype_code(W)
    M, K = W.shape
    if M % R or K % C:
        raise ValueError("M, K must be multiples of R, C")
    indptr = np.zeros(M // R + 1, dtype=np.int32)
    nnzb = lib.ref_bsr_count(_ptr(W), dt, M, K, R, C, threshold, _ptr(indptr))
    if nnzb < 0:
        raise ValueError("bad arguments")
    indices = np.zeros(nnzb, dtype=np.int32)
    data = np.zeros((nnzb, R, C), dtype=W.dtype)
    lib.ref_bsr_fill(_ptr(W), dt, M, K, R, C, threshold, _ptr(indptr), _ptr(indices), _ptr(data))
    return indptr, indices, data


def bsr_to_dense(indptr, indices, data, M: int, K: int) -> np.ndarray:
    lib = _load()
    data = np.ascontiguousarray(data)
    nnzb, R, C = data.shape
    out = np.zeros((M, K), dtype=data.dtype)
    lib.ref_bsr_to_dense(_dtype_code(data), M, K, R, C, _ptr(np.ascontiguousarray(indptr, np.int32)),
                         _ptr(np.ascontiguousarray(indices, np.int32)), _ptr(data), _ptr(out))
    return out


def _apply(fn, indptr, indices, data, X, bias, M, rows):
    lib = _load()
    data = np.ascontiguousarray(data)
    X = np.ascontiguousarray(X)
    if data.dtype != X.dtype:
        raise TypeError("data and X must share a dtype")
    _, R, C = data.shape
    N, K = X.shape
    r, n = _rows(rows, N)
    out = np.zeros((n, M), dtype=np.float64)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    getattr(lib, fn)(_dtype_code(X), M, K, R, C, _ptr(np.ascontiguousarray(indptr, np.int32)),
                     _ptr(np.ascontiguousarray(indices, np.int32)), _ptr(data), _ptr(X), _ptr(b),
                     _ptr(r), n, _ptr(out))
    return out


def bsr_spmm(indptr, indices, data, X, bias, M: int, rows=None) -> np.ndarray:
    """Y = X W^T + b over the stored blocks, float64, for tokens ``rows`` (all if None)."""
    return _apply("ref_bsr_spmm", indptr, indices, data, X, bias, M, rows)


def err_bound(indptr, indices, data, X, bias, M: int, rows=None) -> np.ndarray:
    """sum_k |X[n,k]| |W[m,k]| + |b[m]| for the same tokens."""
    return _apply("ref_bsr_err_bound", indptr, indices, data, X, bias, M, rows)


def bsr_spmm_f32acc(indptr, indices, data, X, bias, M: int, rows=None, threads: int = 1) -> np.ndarray:
    """Y = X W^T + b with a float accumulator (the timed CPU baseline), float32,
    block rows divided among ``threads`` OpenMP threads."""
    lib = _load()
    data = np.ascontiguousarray(data)
    X = np.ascontiguousarray(X)
    if data.dtype != X.dtype:
        raise TypeError("data and X must share a dtype")
    _, R, C = data.shape
    N, K = X.shape
    r, n = _rows(rows, N)
    out = np.zeros((n, M), dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    lib.ref_bsr_spmm_f32acc(_dtype_code(X), M, K, R, C, _ptr(np.ascontiguousarray(indptr, np.int32)),
                            _ptr(np.ascontiguousarray(indices, np.int32)), _ptr(data), _ptr(X), _ptr(b),
                            _ptr(r), n, _ptr(out), int(threads))
    return out


def max_threads() -> int:
    """OpenMP threads the oracle library may use (1 without OpenMP)."""
    return int(_load().ref_max_threads())


def dense_linear(W, X, bias, rows=None) -> np.ndarray:
    lib = _load()
    W = np.ascontiguousarray(W)
    X = np.ascontiguousarray(X)
    M, K = W.shape
    r, n = _rows(rows, X.shape[0])
    out = np.zeros((n, M), dtype=np.float64)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    lib.ref_dense_linear(_dtype_code(X), M, K, _ptr(W), _ptr(X), _ptr(b), _ptr(r), n, _ptr(out))
    return out


def round_f32(Y: np.ndarray) -> np.ndarray:
    Y = np.ascontiguousarray(Y, dtype=np.float64)
    out = np.zeros(Y.shape, dtype=np.float32)
    _load().ref_round_f32(_ptr(Y), _ptr(out), Y.size)
    return out


def round_bf16(Y: np.ndarray) -> np.ndarray:
    """float64 -> bfloat16 bit patterns (uint16), round to nearest even."""
    Y = np.ascontiguousarray(Y, dtype=np.float64)
    out = np.zeros(Y.shape, dtype=np.uint16)
    _load().ref_round_bf16(_ptr(Y), _ptr(out), Y.size)
    return out


def widen(a: np.ndarray) -> np.ndarray:
    """float32 or bf16 bits -> float64 (exact)."""
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return a.astype(np.float64)
