"""bench.py's measurement arithmetic on CPU, against the definitions it
reports: algorithmic bytes of a call (block values, indices, indptr, X, Y and
bias, each once), the unit each kernel kind is held to (FP32 FMA for the SIMT
kernel, the bf16 tensor rate for bf16 MMAs, a third of the tf32 rate for
3xTF32), and the roofline fraction (the slower of FLOPs at that peak and bytes
at HBM bandwidth, over the measured time)."""
from collections import namedtuple

import pytest

import bench
import synth

W = namedtuple("W", "nnz nnzb M K R C dtype")
PK = {"bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "measured"}


def test_call_bytes_of_a_bert_large_weight():
    # 1024x1024 at 90% in 32x1 blocks: 3277 kept blocks (the sparsity reading
    # rounds MB*KB*(100-s)/100 to nearest), 16384 fp32 tokens
    nnzb = synth.kept_blocks(32, 1024, 90)
    assert nnzb == 3277
    w = W(nnzb * 32, nnzb, 1024, 1024, 32, 1, "f32")
    expect = nnzb * 32 * 4 + 4 * nnzb + 4 * (32 + 1) + 16384 * 1024 * 4 * 2 + 4 * 1024
    assert bench.call_bytes(w, 16384, 4) == expect == 134654520


def test_pipe_peaks_per_kernel_kind():
    p, _ = bench.pipe_peak({"variant": "xstage"}, "f32", PK, 78.7)
    assert p == pytest.approx(78.7e12)
    p, _ = bench.pipe_peak({"variant": "tcgen05"}, "bf16", PK, 78.7)
    assert p == pytest.approx(1700e12)
    p, _ = bench.pipe_peak({"variant": "tcgen05"}, "f32", PK, 78.7)
    assert p == pytest.approx(1700e12 * (1.1 / 2.25) / 3)


@pytest.mark.parametrize("variant,us,flops,nbytes,bound", [
    ("xstage", 138.0, 3.44e9, 134.6e6, "alu"),        # 25.5 FLOP/B, above the FP32 ridge
    ("tcgen05", 102.0, 3.44e9, 134.6e6, "hbm"),       # 3xTF32: bytes take longer than FLOPs
])
def test_kernel_roofline_fraction(variant, us, flops, nbytes, bound):
    hbm = 6813.8e9
    peak, desc = bench.pipe_peak({"variant": variant}, "f32", PK, 78.7)
    d = {"ms": 3 * us * 1e-3, "calls": 3, "flops": 3 * flops, "bytes": 3 * nbytes, "peak": peak, "peak_desc": desc,
         "sc": {"variant": variant, "exec_R": 32, "exec_C": 1}, "w": W(0, 0, 1024, 1024, 32, 1, "f32")}
    r = bench.kernel_roofline(d, hbm)
    t = us * 1e-6
    assert r["bound"] == bound
    if bound == "alu":
        assert r["achieved"] == pytest.approx(flops / t / 1e12) and r["unit"] == "TFLOP/s"
    else:
        assert r["achieved"] == pytest.approx(nbytes / t / 1e9) and r["unit"] == "GB/s"
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert r["roofline_frac"] == pytest.approx(max(flops / peak, nbytes / hbm) / t)
    assert r["us_per_launch"] == pytest.approx(us)
