"""Parity sweep of the persistent tensor-core kernel (tcp) on the block
shapes of the tc kernel, for a process started with BSR_TCP=1 (tcp takes
every call of those shapes) and BSR_TC_F32_R16=1 (fp32 16-row blocks on the
tensor cores at any weight size), optionally BSR_TCP_G (one task size). Rows
of every length, a dense row (split into pieces whose fp32 partials the
reduce pass adds), an empty row (bias only), token counts with a ragged last
tile and with several units per CTA, no bias, and a stage that is never
loaded (every wait on it gives up, the call reports BSR_ERR_TIMEOUT and a
later handle still computes correctly). Run by tests/test_gpu_tcp.py in a
subprocess; exit status 0 when every check passes."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

CASES = [  # R, C, dtype, density, N, bias
    (16, 16, "bf16", 0.20, 1000, True), (32, 32, "bf16", 0.25, 777, True), (16, 64, "bf16", 0.20, 5000, False),
    (64, 16, "bf16", 0.20, 300, True), (128, 32, "bf16", 0.20, 1000, True),
    (32, 1, "bf16", 0.30, 1000, True), (1, 1, "bf16", 0.40, 600, True), (4, 4, "bf16", 0.40, 129, True),
    (16, 16, "f32", 0.20, 1000, True), (16, 32, "f32", 0.20, 517, True), (32, 32, "f32", 0.20, 5000, True),
    (64, 16, "f32", 0.20, 128, False),
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
        cnt[1 % MB] = KB     # a dense row
        cnt[MB - 1] = 0      # an empty row: its outputs are the bias
        seed = 6000 + R * 7 + C * 3 + (dt == "bf16")
        w = synth.make_weight("tcp", seed, M, K, R, C, dt, 0, mask=synth.mask_from_row_counts(seed, cnt, KB))
        h = bsr.bsr_create(*build_on_gpu(w.W, R, C), R, C, M, K)
        if h.schedule()["variant"] != "tcgen05":
            print(f"{R}x{C} {dt}: not on the tensor cores ({h.schedule()['variant']})", flush=True)
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
    # a stage that is never loaded: bounded waits, BSR_ERR_TIMEOUT, usable context
    from paper_2106_08846_gb300 import bsrlib as b
    for R, C, dt in ((16, 16, "bf16"), (32, 32, "f32")):
        w = synth.make_weight("tcp_stall", 6100 + R, 256, 512, R, C, dt, 80)
        gpu = build_on_gpu(w.W, R, C)
        os.environ["BSR_WAIT_LIMIT_NS"] = "2000000"
        os.environ["BSR_TEST_STALL_CHUNK"] = "1"
        h = bsr.bsr_create(*gpu, R, C, 256, 512)
        del os.environ["BSR_WAIT_LIMIT_NS"], os.environ["BSR_TEST_STALL_CHUNK"]
        X = synth.activations(6200 + R, 300, 512, dt)
        h.spmm(to_dev(X), to_dev(w.bias))
        torch.cuda.synchronize()
        st = h.check_device_status()
        h2 = bsr.bsr_create(*gpu, R, C, 256, 512)
        Y = to_host(h2.spmm(to_dev(X), to_dev(w.bias)))
        try:
            assert st == b.BSR_ERR_TIMEOUT, st
            assert h2.check_device_status() == b.BSR_OK
            check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, 256)
            print(f"stall {R}x{C} {dt}: ok", flush=True)
        except AssertionError as ex:
            fails += 1
            print(f"stall {R}x{C} {dt}: FAIL {str(ex)[:300]}", flush=True)
    return 1 if fails else 0


if __name__ == "__main__":
    sys.exit(main())
