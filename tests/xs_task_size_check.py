"""Parity sweep of the SIMT kernel at one forced task size, for a process
started with BSR_XS_G (items per CTA): the epilogue differs with the warps
per item (one warp stores its tile from registers, two hand one tile over
through shared memory, more sum slots in an output pass, one-row blocks with
several items per warp). One- and multi-column blocks, fp32 and bf16, rows of
every length, a dense row (split into pieces whose fp32 partials the reduce
pass adds), an empty row (bias only), ragged token counts, no bias. Run by
tests/test_gpu_xs_tasks.py in a subprocess; exit status 0 when every check
passes and at least two cases ran at the forced size."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

CASES = [  # R, C, dtype, density, K, N, bias
    (32, 1, "f32", 0.06, 512, 1000, True), (16, 1, "f32", 0.10, 256, 333, True), (8, 1, "f32", 0.10, 256, 129, False),
    (4, 4, "f32", 0.10, 256, 700, True), (16, 16, "f32", 0.10, 512, 77, True), (2, 1, "f32", 0.10, 256, 64, True),
    (1, 1, "f32", 0.10, 512, 300, True), (1, 32, "f32", 0.20, 512, 65, True), (32, 1, "bf16", 0.05, 512, 1000, True),
    (1, 1, "bf16", 0.02, 512, 129, False),
]


def main() -> int:
    import torch

    import oracle
    import synth
    import paper_2106_08846_gb300 as bsr
    from tests.gpu_util import build_on_gpu, check_product, to_dev, to_host
    G = int(os.environ["BSR_XS_G"])
    fails = ran = 0
    for R, C, dt, dens, K, N, with_bias in CASES:
        if G > 14 and R != 1:   # several items per warp: one-row blocks only
            continue
        M = 384
        MB, KB = M // R, K // C
        cnt = np.full(MB, max(1, int(round(KB * dens))), dtype=np.int64)
        cnt[1 % MB] = KB     # a dense row
        cnt[MB - 1] = 0      # an empty row: its outputs are the bias
        seed = 8000 + R * 7 + C * 3 + K + (dt == "bf16")
        w = synth.make_weight("xsg", seed, M, K, R, C, dt, 0, mask=synth.mask_from_row_counts(seed, cnt, KB))
        h = bsr.bsr_create(*build_on_gpu(w.W, R, C), R, C, M, K)
        if h.schedule()["variant"] != "xstage":
            print(f"{R}x{C} {dt}: not on the SIMT kernel ({h.schedule()['variant']})", flush=True)
            fails += 1
            continue
        sizes = str(h.schedule()["xstage_task_sizes"]).split(",")
        forced = str(G) in sizes
        ran += forced
        X = synth.activations(seed + 1, N, K, dt)
        b = w.bias if with_bias else None
        Y = h.spmm(to_dev(X), to_dev(b) if with_bias else None)
        torch.cuda.synchronize()
        try:
            assert h.check_device_status() == 0
            e = check_product(to_host(Y), oracle.bsr_from_dense(w.W, R, C), X, b, M)
            how = f"G={G}" if forced else f"G={G} does not fit, chosen per call"
            print(f"{R}x{C} {dt} N={N} {how}: ok (max scaled error {e:.3g})", flush=True)
        except AssertionError as ex:
            fails += 1
            print(f"{R}x{C} {dt} N={N} G={G}: FAIL {str(ex)[:300]}", flush=True)
        h.destroy()
    if ran < 2:
        print(f"only {ran} cases ran at G={G}", flush=True)
        fails += 1
    return 1 if fails else 0


if __name__ == "__main__":
    sys.exit(main())
