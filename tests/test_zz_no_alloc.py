"""bsr_spmm_noalloc, the entry point for callers that cannot allocate device
memory (graph capture, fixed budgets, no implicit synchronisation): it must
give the same product as bsr_spmm, call after call, through the fixed scratch
array, and refuse work that does not fit the array. This file is collected
last so that a failure here comes after every other test has run."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import build_on_gpu, check_product, to_dev, to_host

pytestmark = pytest.mark.gpu


def _split_weight(R, C, dtype, seed):
    # a few fully dense block rows among short and empty ones: split rows,
    # so the partial tiles go through the scratch array
    M, K = 512, 2048
    MB, KB = M // R, K // C
    cnt = np.zeros(MB, dtype=np.int64)
    cnt[1::2] = 2
    cnt[[3, MB // 2, MB - 2]] = KB
    return synth.make_weight("na", seed, M, K, R, C, dtype, 0, mask=synth.mask_from_row_counts(seed, cnt, KB))


@pytest.mark.parametrize("R,C,dtype", [(32, 1, "f32"), (16, 16, "bf16"), (8, 1, "f32")])
def test_noalloc_matches_bsr_spmm_twice(R, C, dtype):
    import paper_2106_08846_gb300 as bsr
    w = _split_weight(R, C, dtype, 5000 + R + C)
    gpu = build_on_gpu(w.W, R, C)
    h = bsr.bsr_create(*gpu, R, C, w.M, w.K)
    assert h.schedule()["slots"] > 0
    X = synth.activations(5100 + R, 300, w.K, dtype)
    Xd, bd = to_dev(X), to_dev(w.bias)
    Y_ref = torch.empty((300, w.M), dtype=Xd.dtype, device="cuda")
    bsr.bsr_spmm(h, Xd, bd, Y_ref, 300)
    ref = oracle.bsr_from_dense(w.W, R, C)
    for _ in range(2):
        Y = torch.full((300, w.M), float("nan"), dtype=Xd.dtype, device="cuda")
        bsr.bsr_spmm_noalloc(h, Xd, bd, Y, 300)
        torch.cuda.synchronize()
        assert h.check_device_status() == 0
        got, want = to_host(Y), to_host(Y_ref)
        # same tolerance as every product test, against the oracle and against bsr_spmm
        check_product(got, ref, X, w.bias, w.M)
        tol = 1e-5 if dtype == "f32" else 1e-2
        E = oracle.err_bound(*ref, X, w.bias, w.M)
        assert np.all(np.abs(oracle.widen(got) - oracle.widen(want)) <= tol * E)


def test_noalloc_rejects_oversized_and_host_buffers():
    import paper_2106_08846_gb300 as bsr
    from paper_2106_08846_gb300 import bsrlib
    w = _split_weight(32, 1, "f32", 5200)
    h = bsr.bsr_create(*build_on_gpu(w.W, 32, 1), 32, 1, w.M, w.K)
    sched = h.schedule()
    limit = 32 << 20
    n_big = limit // (sched["slots"] * sched["exec_R"] * 4) + 1
    X = torch.zeros((8, w.K), device="cuda")
    Y = torch.zeros((8, w.M), device="cuda")
    lib = bsr.load()
    import ctypes
    P = ctypes.c_void_p
    # oversized: rejected before anything is launched
    assert lib.bsr_spmm_noalloc(h.ptr, P(X.data_ptr()), None, P(Y.data_ptr()), n_big, None) == bsrlib.BSR_ERR_CAPACITY
    # host buffers need staging memory: refused
    Xh = torch.zeros((8, w.K)).pin_memory()
    Yh = torch.zeros((8, w.M)).pin_memory()
    assert lib.bsr_spmm_noalloc(h.ptr, P(Xh.data_ptr()), None, P(Yh.data_ptr()), 8, None) == bsrlib.BSR_ERR_INVALID_ARG
    assert h.check_device_status() == 0


def test_noalloc_capacity_counts_the_executed_block_height():
    # 1x32 bf16 blocks dense enough to run on the tensor cores as zero-filled
    # 16 x 64 tiles: the scratch a call needs is slots * N * exec_R * 4 bytes
    # (exec_R = 16, not R = 1). N at the limit runs and equals bsr_spmm; one
    # token more is refused before anything is launched.
    import ctypes

    import paper_2106_08846_gb300 as bsr
    from paper_2106_08846_gb300 import bsrlib
    R, C, M, K = 1, 32, 256, 8192
    MB, KB = M // R, K // C
    cnt = np.full(MB, 2, dtype=np.int64)
    cnt[:32] = KB   # two fully dense tile rows, split across CTAs
    w = synth.make_weight("na_rb", 5300, M, K, R, C, "bf16", 0, mask=synth.mask_from_row_counts(5300, cnt, KB))
    h = bsr.bsr_create(*build_on_gpu(w.W, R, C), R, C, M, K)
    sc = h.schedule()
    assert sc["variant"] == "tcgen05" and sc["exec_R"] == 16 and sc["R"] == 1 and sc["slots"] > 0
    n_max = (32 << 20) // (sc["slots"] * sc["exec_R"] * 4)
    g = torch.Generator(device="cuda").manual_seed(5301)
    X = torch.randn((n_max + 1, K), generator=g, device="cuda").to(torch.bfloat16)
    bd = to_dev(w.bias)
    Y = torch.empty((n_max + 1, M), dtype=torch.bfloat16, device="cuda")
    Y_ref = torch.empty((n_max, M), dtype=torch.bfloat16, device="cuda")
    lib = bsr.load()
    P = ctypes.c_void_p
    assert lib.bsr_spmm_noalloc(h.ptr, P(X.data_ptr()), P(bd.data_ptr()), P(Y.data_ptr()), n_max + 1,
                                None) == bsrlib.BSR_ERR_CAPACITY
    bsr.bsr_spmm_noalloc(h, X[:n_max], bd, Y[:n_max], n_max)
    bsr.bsr_spmm(h, X[:n_max], bd, Y_ref, n_max)
    torch.cuda.synchronize()
    assert h.check_device_status() == 0
    assert torch.equal(Y[:n_max].view(torch.int16), Y_ref.view(torch.int16))
    # and a sample of tokens against the oracle
    rows = np.array([0, 1, n_max // 2, n_max - 1])
    check_product(to_host(Y[:n_max])[rows], oracle.bsr_from_dense(w.W, R, C), to_host(X[rows]), w.bias, M)
    h.destroy()
