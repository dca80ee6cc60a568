"""Parity sweep of the gathered-K tensor-core kernel on every block shape it
runs, for a process started with BSR_GK=1 (the kernel takes every call of a
shape it supports) and optionally BSR_GK_G (one task size). Run by
tests/test_gpu_gk.py in a subprocess; exit status 0 when every output element
is within the fp32 / bf16 tolerance of the oracle."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

CASES = [  # R, C, dtype, density, N, bias
    (32, 1, "f32", 0.10, 1000, True), (16, 1, "f32", 0.10, 700, True), (16, 16, "f32", 0.20, 600, True),
    (32, 32, "f32", 0.20, 1000, False), (64, 4, "f32", 0.20, 517, True), (128, 2, "f32", 0.10, 1000, True),
    (16, 8, "f32", 0.20, 640, True), (32, 2, "f32", 0.20, 1000, True),
    (32, 1, "bf16", 0.10, 1000, True), (16, 16, "bf16", 0.20, 777, True), (32, 32, "bf16", 0.20, 1000, True),
    (16, 2, "bf16", 0.15, 1000, False), (64, 8, "bf16", 0.20, 530, True), (128, 1, "bf16", 0.05, 1000, True),
    (32, 4, "bf16", 0.20, 1000, True),
]


def main() -> int:
    import torch

    import oracle
    import synth
    import paper_2106_08846_gb300 as bsr
    from tests.gpu_util import build_on_gpu, check_product, to_dev, to_host
    fails = 0
    for R, C, dt, dens, N, with_bias in CASES:
        M, K = 512, 768
        MB, KB = M // R, K // C
        cnt = np.full(MB, max(1, int(round(KB * dens))), dtype=np.int64)
        cnt[1] = KB          # a dense row: entries split into several pieces
        cnt[MB - 1] = 0      # an empty row: its outputs are the bias
        seed = 4000 + R * 7 + C * 3 + (dt == "bf16")
        w = synth.make_weight("gk", seed, M, K, R, C, dt, 0, mask=synth.mask_from_row_counts(seed, cnt, KB))
        h = bsr.bsr_create(*build_on_gpu(w.W, R, C), R, C, M, K)
        if h.schedule()["gk_task_sizes"] == "none":
            print(f"{R}x{C} {dt}: the kernel does not fit", flush=True)
            fails += 1
            continue
        X = synth.activations(seed + 1, N, K, dt)
        b = w.bias if with_bias else None
        Y = h.spmm(to_dev(X), to_dev(b) if with_bias else None)
        torch.cuda.synchronize()
        try:
            assert h.check_device_status() == 0
            e = check_product(to_host(Y), oracle.bsr_from_dense(w.W, R, C), X, b, M)
            print(f"{R}x{C} {dt} N={N}: ok (max scaled error {e:.3g})", flush=True)
        except AssertionError as ex:
            fails += 1
            print(f"{R}x{C} {dt} N={N}: FAIL {str(ex)[:300]}", flush=True)
        h.destroy()
    return 1 if fails else 0


if __name__ == "__main__":
    sys.exit(main())
