"""Helpers for the GPU tests: move generator output to the device, run the C ABI
through the binding, and compare with the CPU oracle element by element."""
import numpy as np
import torch

import oracle

TOL = {"f32": 1e-5, "bf16": 1e-2}


def dtype_of(a: np.ndarray) -> str:
    return "bf16" if a.dtype == np.uint16 else "f32"


def to_dev(a: np.ndarray, dev="cuda") -> torch.Tensor:
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev)
    return torch.from_numpy(a).to(dev)


def to_host(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def as_f64(a: np.ndarray) -> np.ndarray:
    return oracle.widen(a)


def build_on_gpu(W: np.ndarray, R: int, C: int, thr: float = 0.0):
    import paper_2106_08846_gb300 as bsr
    return bsr.bsr_from_dense(to_dev(W), R, C, thr)


def assert_structure_equal(gpu, ref):
    indptr, indices, data = (to_host(t) for t in gpu)
    assert np.array_equal(indptr, ref[0]), "indptr"
    assert np.array_equal(indices, ref[1]), "indices"
    assert data.shape == ref[2].shape
    assert data.tobytes() == np.ascontiguousarray(ref[2]).tobytes(), "data bits"


def check_product(Y_gpu: np.ndarray, ref_bsr, X: np.ndarray, bias, M: int, rows=None, tol=None):
    """|Y_gpu - Y_oracle| <= tol * (sum |x||w| + |b|) elementwise, tokens `rows`."""
    dt = dtype_of(X)
    tol = TOL[dt] if tol is None else tol
    Yr = oracle.bsr_spmm(*ref_bsr, X, bias, M, rows=rows)
    E = oracle.err_bound(*ref_bsr, X, bias, M, rows=rows)
    got = as_f64(Y_gpu if rows is None else Y_gpu[np.asarray(rows)])
    assert got.shape == Yr.shape
    assert np.all(np.isfinite(got))
    err = np.abs(got - Yr)
    bad = err > tol * E
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{bad.sum()} of {bad.size} outside tolerance; first at {tuple(i)}: "
                             f"gpu={got[tuple(i)]!r} ref={Yr[tuple(i)]!r} bound={tol * E[tuple(i)]!r}")
    return float((err / np.maximum(E, 1e-300)).max())
