"""Property test of the whole GPU path on random tiny shapes: seeded cases
with M, K <= 64 (and a few up to 128 so the tensor-core shapes appear), a
block shape (R, C) dividing them, block sparsity from 0% to 100%, 1 to 200
tokens, with or without bias. Every case runs the C ABI -- bsr_from_dense
(bit-exact against the oracle), bsr_create, bsr_spmm -- and compares every
output with the oracle at the fp32 / bf16 tolerance, whichever kernel the
schedule picks (SIMT, tensor-core tiles, generic)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import assert_structure_equal, build_on_gpu, check_product, to_dev, to_host

pytestmark = pytest.mark.gpu


def _divisors(n):
    return [d for d in range(1, n + 1) if n % d == 0]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_gpu_random_tiny_shapes(dtype):
    import paper_2106_08846_gb300 as bsr
    rng = np.random.default_rng(7106 + (dtype == "bf16"))
    variants = set()
    for case in range(50):
        big = case % 5 == 0
        M = int(rng.choice([32, 64, 96, 128])) if big else int(rng.integers(1, 65))
        K = int(rng.choice([32, 64, 96, 128])) if big else int(rng.integers(1, 65))
        R, C = int(rng.choice(_divisors(M))), int(rng.choice(_divisors(K)))
        MB, KB = M // R, K // C
        nnzb = int(round(MB * KB * float(rng.choice([0.0, 0.15, 0.4, 0.8, 1.0]))))
        mask = synth.uniform_block_mask(8000 + case, MB, KB, nnzb)
        W = synth.weight_values(8000 + case, mask, R, C)
        if dtype == "bf16":
            W = synth.to_bf16_bits(W)
        N = int(rng.integers(1, 201))
        X = synth.activations(9000 + case, N, K, dtype)
        b = synth.normal(9500 + case, 0, M, 0.02).astype(np.float32) if case % 3 else None
        ref = oracle.bsr_from_dense(W, R, C)
        gpu = build_on_gpu(W, R, C)
        assert_structure_equal(gpu, ref)
        h = bsr.bsr_create(*gpu, R, C, M, K)
        variants.add(h.schedule()["variant"])
        Y = h.spmm(to_dev(X), None if b is None else to_dev(b))
        torch.cuda.synchronize()
        assert h.check_device_status() == 0, (case, M, K, R, C)
        check_product(to_host(Y), ref, X, b, M)
        h.destroy()
    assert {"xstage", "generic"} <= variants
