"""ctypes binding of include/bsr.h, with the same names.

Argument marshalling only: every step of the product and of the BSR
conversion runs in libbsr_gb300.so. torch supplies device memory, streams and
tensors; tensors cross as ``data_ptr()`` and streams as their ``cuda_stream``.
There is no CPU fallback: if the library is missing, loading raises.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libbsr_gb300.so")

BSR_OK = 0
BSR_ERR_INVALID_ARG = 1
BSR_ERR_SHAPE = 2
BSR_ERR_UNSUPPORTED = 3
BSR_ERR_CAPACITY = 4
BSR_ERR_STRUCTURE = 5
BSR_ERR_ALIGNMENT = 6
BSR_ERR_CUDA = 7
BSR_ERR_TIMEOUT = 8
BSR_ERR_ALLOC = 9

BSR_F32 = 0
BSR_BF16 = 1

_DT = {torch.float32: BSR_F32, torch.bfloat16: BSR_BF16}
_TORCH_DT = {BSR_F32: torch.float32, BSR_BF16: torch.bfloat16}

_lib = None


class BsrError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {bsr_status_str(status)}")


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libbsr_gb300.so (built by ``__graft_entry__.build()``); raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build the CUDA library first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(path)
        P, I64, I, U = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_int
        lib.bsr_from_dense.argtypes = [P, I64, I64, I, I, ctypes.c_float, U, P, P, P, I64,
                                       ctypes.POINTER(I64), P]
        lib.bsr_from_dense.restype = U
        lib.bsr_create.argtypes = [P, P, P, I, I, I64, I64, U, ctypes.POINTER(P)]
        lib.bsr_create.restype = U
        lib.bsr_reserve.argtypes = [P, I64]
        lib.bsr_reserve.restype = U
        lib.bsr_spmm.argtypes = [P, P, P, P, I64, P]
        lib.bsr_spmm.restype = U
        lib.bsr_spmm_noalloc.argtypes = [P, P, P, P, I64, P]
        lib.bsr_spmm_noalloc.restype = U
        lib.bsr_spmm_batch.argtypes = [ctypes.POINTER(P), ctypes.c_int, P, ctypes.POINTER(P), ctypes.POINTER(P),
                                       I64, P]
        lib.bsr_spmm_batch.restype = U
        lib.bsr_plan_create.argtypes = [ctypes.POINTER(P), ctypes.POINTER(P), ctypes.POINTER(P), ctypes.POINTER(P),
                                        ctypes.POINTER(I64), ctypes.c_int, ctypes.c_int, ctypes.POINTER(P)]
        lib.bsr_plan_create.restype = U
        lib.bsr_plan_launch.argtypes = [P, P]
        lib.bsr_plan_launch.restype = U
        lib.bsr_plan_get_order.argtypes = [P, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int), ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_int)]
        lib.bsr_plan_get_order.restype = U
        lib.bsr_plan_destroy.argtypes = [P]
        lib.bsr_plan_destroy.restype = None
        lib.bsr_check_device_status.argtypes = [P]
        lib.bsr_check_device_status.restype = U
        lib.bsr_get_schedule.argtypes = [P, ctypes.c_char_p, ctypes.c_size_t]
        lib.bsr_get_schedule.restype = U
        lib.bsr_destroy.argtypes = [P]
        lib.bsr_destroy.restype = None
        lib.bsr_status_str.argtypes = [U]
        lib.bsr_status_str.restype = ctypes.c_char_p
        _lib = lib
    return _lib


def bsr_status_str(status: int) -> str:
    return load().bsr_status_str(status).decode()


def _check(status: int, where: str) -> None:
    if status != BSR_OK:
        raise BsrError(status, where)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def dtype_code(dtype: torch.dtype) -> int:
    if dtype not in _DT:
        raise TypeError(f"unsupported dtype {dtype}: float32 or bfloat16")
    return _DT[dtype]


def bsr_from_dense(W: torch.Tensor, R: int, C: int, threshold: float = 0.0, stream=None
                   ) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """BSR arrays (indptr, indices, data[nnzb, R, C]) of the dense device weight W[M, K].

    Two calls of the C function: a query for nnzb, then the fill into
    tensors allocated here.
    """
    lib = load()
    if not W.is_cuda or not W.is_contiguous():
        raise ValueError("W must be a contiguous CUDA tensor")
    M, K = W.shape
    dt = dtype_code(W.dtype)
    if R <= 0 or C <= 0 or M % R or K % C:
        _check(BSR_ERR_SHAPE, "bsr_from_dense")
    indptr = torch.empty(M // R + 1, dtype=torch.int32, device=W.device)
    nnzb = ctypes.c_int64(0)
    s = _stream(stream)
    _check(lib.bsr_from_dense(_ptr(W), M, K, R, C, threshold, dt, _ptr(indptr), None, None, 0,
                              ctypes.byref(nnzb), s), "bsr_from_dense(query)")
    n = nnzb.value
    indices = torch.empty(max(n, 0), dtype=torch.int32, device=W.device)
    data = torch.empty((max(n, 0), R, C), dtype=W.dtype, device=W.device)
    if n > 0:
        _check(lib.bsr_from_dense(_ptr(W), M, K, R, C, threshold, dt, _ptr(indptr), _ptr(indices),
                                  _ptr(data), n, ctypes.byref(nnzb), s), "bsr_from_dense")
    return indptr, indices, data


class Handle:
    """A created BSR operator. Keeps its borrowed arrays alive until destroyed."""

    def __init__(self, ptr: ctypes.c_void_p, arrays, R, C, M, K, dtype):
        self._ptr = ptr
        self._arrays = arrays
        self.R, self.C, self.M, self.K, self.dtype = R, C, M, K, dtype

    @property
    def ptr(self) -> ctypes.c_void_p:
        if self._ptr is None:
            raise RuntimeError("handle destroyed")
        return self._ptr

    def spmm(self, X: torch.Tensor, bias: Optional[torch.Tensor] = None, Y: Optional[torch.Tensor] = None,
             stream=None) -> torch.Tensor:
        if Y is None:
            Y = torch.empty((X.shape[0], self.M), dtype=X.dtype, device=X.device,
                            pin_memory=not X.is_cuda)
        bsr_spmm(self, X, bias, Y, X.shape[0], stream)
        return Y

    def reserve(self, N_max: int) -> None:
        bsr_reserve(self, N_max)

    def schedule(self) -> dict:
        return parse_schedule(bsr_get_schedule(self))

    def check_device_status(self) -> int:
        return bsr_check_device_status(self)

    def destroy(self) -> None:
        if self._ptr is not None:
            load().bsr_destroy(self._ptr)
            self._ptr = None
            self._arrays = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def bsr_create(indptr: torch.Tensor, indices: torch.Tensor, data: torch.Tensor, R: int, C: int,
               M: int, K: int) -> Handle:
    lib = load()
    for name, t in (("indptr", indptr), ("indices", indices), ("data", data)):
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
    if indptr.dtype != torch.int32 or indices.dtype != torch.int32:
        raise TypeError("indptr and indices must be int32")
    out = ctypes.c_void_p()
    _check(lib.bsr_create(_ptr(indptr), _ptr(indices) if indices.numel() else None,
                          _ptr(data) if data.numel() else None, R, C, M, K, dtype_code(data.dtype),
                          ctypes.byref(out)), "bsr_create")
    return Handle(out, (indptr, indices, data), R, C, M, K, data.dtype)


def bsr_reserve(h: Handle, N_max: int) -> None:
    _check(load().bsr_reserve(h.ptr, N_max), "bsr_reserve")


def bsr_spmm(h: Handle, X: torch.Tensor, bias: Optional[torch.Tensor], Y: torch.Tensor,
             N: Optional[int] = None, stream=None) -> None:
    """Y[N, M] = X[N, K] W^T + bias; X and Y both on the device or both in host memory."""
    if X.dtype != h.dtype or Y.dtype != h.dtype:
        raise TypeError("X and Y must have the handle's dtype")
    if not X.is_contiguous() or not Y.is_contiguous():
        raise ValueError("X and Y must be contiguous")
    if bias is not None and (bias.dtype != torch.float32 or not bias.is_contiguous()):
        raise TypeError("bias must be a contiguous float32 tensor")
    N = X.shape[0] if N is None else N
    if X.shape[-1] != h.K or Y.shape[-1] != h.M or X.shape[0] < N or Y.shape[0] < N:
        raise ValueError("X must be [N, K] and Y [N, M]")
    _check(load().bsr_spmm(h.ptr, _ptr(X), _ptr(bias), _ptr(Y), N, _stream(stream)), "bsr_spmm")


def bsr_spmm_noalloc(h: Handle, X: torch.Tensor, bias: Optional[torch.Tensor], Y: torch.Tensor,
                     N: Optional[int] = None, stream=None) -> None:
    """bsr_spmm without any device allocation (device X and Y only): split-row
    partials use the library's fixed scratch array (see include/bsr.h)."""
    if X.dtype != h.dtype or Y.dtype != h.dtype:
        raise TypeError("X and Y must have the handle's dtype")
    if not X.is_contiguous() or not Y.is_contiguous():
        raise ValueError("X and Y must be contiguous")
    if bias is not None and (bias.dtype != torch.float32 or not bias.is_contiguous()):
        raise TypeError("bias must be a contiguous float32 tensor")
    N = X.shape[0] if N is None else N
    if X.shape[-1] != h.K or Y.shape[-1] != h.M or X.shape[0] < N or Y.shape[0] < N:
        raise ValueError("X must be [N, K] and Y [N, M]")
    _check(load().bsr_spmm_noalloc(h.ptr, _ptr(X), _ptr(bias), _ptr(Y), N, _stream(stream)), "bsr_spmm_noalloc")


def bsr_spmm_batch(handles, X: torch.Tensor, biases, Ys, N: Optional[int] = None, stream=None) -> None:
    """Ys[i][N, M_i] = X[N, K] W_i^T + biases[i] for handles sharing X (device
    tensors only); fused products run as one grid (see include/bsr.h)."""
    n = len(handles)
    if len(Ys) != n or (biases is not None and len(biases) != n):
        raise ValueError("one output (and bias, if given) per handle")
    if not X.is_contiguous():
        raise ValueError("X must be contiguous")
    N = X.shape[0] if N is None else N
    if n and (X.shape[-1] != handles[0].K or X.shape[0] < N):
        raise ValueError("X must be [N, K]")   # (a K that differs between handles: BSR_ERR_SHAPE)
    for h, Y in zip(handles, Ys):
        if X.dtype != h.dtype or Y.dtype != h.dtype:
            raise TypeError("X and every Y must have the handles' dtype")
        if not Y.is_contiguous() or Y.shape[-1] != h.M or Y.shape[0] < N:
            raise ValueError("each Y must be [N, M] and contiguous")
    if biases is not None:
        for b in biases:
            if b is not None and (b.dtype != torch.float32 or not b.is_contiguous()):
                raise TypeError("biases must be contiguous float32 tensors")
    P = ctypes.c_void_p
    harr = (P * max(n, 1))(*[h.ptr for h in handles])
    yarr = (P * max(n, 1))(*[_ptr(Y) for Y in Ys])
    barr = None if biases is None else (P * max(n, 1))(*[_ptr(b) for b in biases])
    _check(load().bsr_spmm_batch(harr, n, _ptr(X), barr, yarr, N, _stream(stream)), "bsr_spmm_batch")


class Plan:
    """A product sequence captured into a CUDA graph (bsr_plan_create). Keeps
    the handles and tensors it was built on alive."""

    def __init__(self, ptr, n, keep):
        self._ptr = ptr
        self.n = n
        self._keep = keep

    def launch(self, stream=None) -> None:
        _check(load().bsr_plan_launch(self._ptr, _stream(stream)), "bsr_plan_launch")

    def order(self):
        """(order, call, n_kernels): the product executed k-th, the library call
        that runs it, and the kernel launches in the graph."""
        n = max(self.n, 1)
        o, c, k = (ctypes.c_int * n)(), (ctypes.c_int * n)(), ctypes.c_int(0)
        _check(load().bsr_plan_get_order(self._ptr, o, c, self.n, ctypes.byref(k)), "bsr_plan_get_order")
        run = [i for i in range(self.n) if o[i] >= 0]
        return [o[i] for i in run], [c[i] for i in run], k.value

    def destroy(self) -> None:
        if self._ptr is not None:
            load().bsr_plan_destroy(self._ptr)
            self._ptr = None
            self._keep = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def bsr_plan_create(handles, Xs, biases, Ys, Ns=None, independent: bool = False) -> Plan:
    """Captures the products Ys[i] = Xs[i] W_i^T + biases[i] (device tensors)
    into one CUDA graph; with ``independent`` the plan may regroup and fuse
    them (see include/bsr.h)."""
    n = len(handles)
    if len(Xs) != n or len(Ys) != n or (biases is not None and len(biases) != n):
        raise ValueError("one X, Y (and bias, if given) per handle")
    Ns = [X.shape[0] for X in Xs] if Ns is None else list(Ns)
    for h, X, Y, N in zip(handles, Xs, Ys, Ns):
        if X.dtype != h.dtype or Y.dtype != h.dtype:
            raise TypeError("X and Y must have the handle's dtype")
        if not X.is_contiguous() or not Y.is_contiguous():
            raise ValueError("X and Y must be contiguous")
        if X.shape[-1] != h.K or Y.shape[-1] != h.M or X.shape[0] < N or Y.shape[0] < N:
            raise ValueError("X must be [N, K] and Y [N, M]")
    if biases is not None:
        for b in biases:
            if b is not None and (b.dtype != torch.float32 or not b.is_contiguous()):
                raise TypeError("biases must be contiguous float32 tensors")
    P = ctypes.c_void_p
    m = max(n, 1)
    harr = (P * m)(*[h.ptr for h in handles])
    xarr = (P * m)(*[_ptr(X) for X in Xs])
    yarr = (P * m)(*[_ptr(Y) for Y in Ys])
    barr = None if biases is None else (P * m)(*[_ptr(b) for b in biases])
    narr = (ctypes.c_int64 * m)(*Ns)
    out = P()
    _check(load().bsr_plan_create(harr, xarr, barr, yarr, narr, n, int(bool(independent)), ctypes.byref(out)),
           "bsr_plan_create")
    return Plan(out, n, (list(handles), list(Xs), list(Ys), None if biases is None else list(biases)))


def bsr_check_device_status(h: Handle) -> int:
    return load().bsr_check_device_status(h.ptr)


def bsr_get_schedule(h: Handle) -> str:
    buf = ctypes.create_string_buffer(4096)
    _check(load().bsr_get_schedule(h.ptr, buf, len(buf)), "bsr_get_schedule")
    return buf.value.decode()


def bsr_destroy(h: Handle) -> None:
    h.destroy()


def parse_schedule(text: str) -> dict:
    out = {}
    for line in text.splitlines():
        m = re.match(r"^(\w+)=(.*)$", line)
        if m:
            k, v = m.groups()
            try:
                out[k] = int(v)
            except ValueError:
                out[k] = v
    return out
