"""bsr_spmm_batch: several products that share X in one call.

Products of one kernel template run as one fused grid; the result of each
must be bit-identical to a bsr_spmm call with the same arguments (the fused
grid runs the same CTAs with the same arguments) and within the tolerance of
the oracle (Section 2.2's product)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import build_on_gpu, check_product, to_dev, to_host

pytestmark = pytest.mark.gpu


def _bsr():
    import paper_2106_08846_gb300 as bsr
    return bsr


def _weight(seed, M, K, R, C, dtype, density, long_rows=()):
    MB, KB = M // R, K // C
    if long_rows:
        cnt = np.full(MB, max(1, int(KB * density)), dtype=np.int64)
        cnt[list(long_rows)] = KB
        mask = synth.mask_from_row_counts(seed, cnt, KB)
    else:
        mask = synth.uniform_block_mask(seed, MB, KB, max(1, int(round(MB * KB * density))))
    return synth.make_weight("b", seed, M, K, R, C, dtype, 0, mask=mask)


def _handles(ws, N):
    bsr = _bsr()
    hs = []
    for w in ws:
        h = bsr.bsr_create(*build_on_gpu(w.W, w.R, w.C), w.R, w.C, w.M, w.K)
        h.reserve(N)
        hs.append(h)
    return hs


def _run_both(ws, N, dtype, seed, with_bias=True):
    bsr = _bsr()
    hs = _handles(ws, N)
    X = synth.activations(seed, N, ws[0].K, dtype)
    Xd = to_dev(X)
    bs = [to_dev(w.bias) for w in ws] if with_bias else None
    Yb = [torch.empty((N, w.M), device="cuda", dtype=Xd.dtype) for w in ws]
    bsr.bsr_spmm_batch(hs, Xd, bs, Yb, N)
    Ys = []
    for i, (h, w) in enumerate(zip(hs, ws)):
        Y = torch.empty((N, w.M), device="cuda", dtype=Xd.dtype)
        bsr.bsr_spmm(h, Xd, bs[i] if bs else None, Y, N)
        Ys.append(Y)
    torch.cuda.synchronize()
    for h in hs:
        assert h.check_device_status() == 0
    return hs, X, [to_host(y) for y in Yb], [to_host(y) for y in Ys]


DENSE, SPARSE = (0.5, 0.3, 0.2), (0.06, 0.04, 0.02)   # SPARSE: bf16 narrow blocks stay SIMT below 1/12 fill


@pytest.mark.parametrize("R,C,dtype,dens,kind", [(32, 1, "f32", DENSE, "xstage"), (1, 1, "f32", DENSE, "xstage"),
                                                 (16, 16, "f32", DENSE, "xstage"), (4, 4, "f32", DENSE, "xstage"),
                                                 (1, 1, "bf16", SPARSE, "xstage"), (8, 1, "bf16", SPARSE, "xstage"),
                                                 (1, 1, "bf16", DENSE, "tcgen05"), (16, 16, "bf16", DENSE, "tcgen05"),
                                                 (32, 32, "bf16", DENSE, "tcgen05"), (32, 32, "f32", DENSE, "tcgen05")])
def test_batch_matches_single_calls_bitwise_and_oracle(R, C, dtype, dens, kind):
    """Three weights of one shape (a query/key/value triple) at different
    sparsities: one fused grid, outputs equal to separate calls bit for bit."""
    N = 200
    ws = [_weight(1500 + 10 * i + R + C, 512, 384, R, C, dtype, d) for i, d in enumerate(dens)]
    hs, X, Yb, Ys = _run_both(ws, N, dtype, 1599)
    assert all(h.schedule()["variant"] == kind for h in hs)
    for w, yb, ys in zip(ws, Yb, Ys):
        assert np.array_equal(yb.view(np.uint8), ys.view(np.uint8))
        check_product(yb, oracle.bsr_from_dense(w.W, w.R, w.C), X, w.bias, w.M)


def test_batch_mixed_kernels_split_rows_and_no_bias():
    """Mixed shapes and kernels in one call (a fused xstage group, a fused
    tensor-core group, a generic product), a weight with split rows (workspace
    and reduce pass after the fused grid), different M per weight, no biases."""
    N = 333
    ws = [
        _weight(1601, 256, 512, 32, 1, "f32", 0.2),
        _weight(1602, 512, 512, 32, 32, "f32", 0.3),                     # tensor cores
        _weight(1603, 384, 512, 32, 1, "f32", 0.05, long_rows=(2, 5)),   # split rows
        _weight(1604, 255, 512, 3, 2, "f32", 0.2),                       # generic kernel
        _weight(1605, 768, 512, 32, 1, "f32", 0.1),
        _weight(1606, 256, 512, 32, 32, "f32", 0.05, long_rows=(1,)),    # tensor cores, one long row
    ]
    hs, X, Yb, Ys = _run_both(ws, N, "f32", 1607, with_bias=False)
    kinds = [h.schedule()["variant"] for h in hs]
    assert kinds == ["xstage", "tcgen05", "xstage", "generic", "xstage", "tcgen05"]
    assert hs[2].schedule()["split_rows"] >= 1
    for w, yb, ys in zip(ws, Yb, Ys):
        assert np.array_equal(yb, ys)
        check_product(yb, oracle.bsr_from_dense(w.W, w.R, w.C), X, None, w.M)


def test_batch_more_products_than_one_grid_holds():
    """70 products of one shape: the call splits them into fused grids of at
    most 64; every output matches its single call."""
    bsr = _bsr()
    N, M, K = 96, 64, 128
    ws = [_weight(1700 + i, M, K, 8, 1, "f32", 0.1 + 0.01 * (i % 7)) for i in range(70)]
    hs = _handles(ws, N)
    X = synth.activations(1799, N, K, "f32")
    Xd = to_dev(X)
    Yb = [torch.empty((N, M), device="cuda") for _ in ws]
    bsr.bsr_spmm_batch(hs, Xd, None, Yb, N)
    torch.cuda.synchronize()
    for i in (0, 33, 63, 64, 69):
        Y = torch.empty((N, M), device="cuda")
        bsr.bsr_spmm(hs[i], Xd, None, Y, N)
        torch.cuda.synchronize()
        assert np.array_equal(to_host(Yb[i]), to_host(Y)), i
    for i in (5, 66):
        check_product(to_host(Yb[i]), oracle.bsr_from_dense(ws[i].W, 8, 1), X, None, M)


def test_batch_argument_errors():
    bsr = _bsr()
    N = 64
    w1 = _weight(1801, 128, 256, 8, 1, "f32", 0.2)
    w2 = _weight(1802, 128, 128, 8, 1, "f32", 0.2)
    h1, h2 = _handles([w1, w2], N)
    X = to_dev(synth.activations(1803, N, 256, "f32"))
    Y1, Y2 = torch.empty((N, 128), device="cuda"), torch.empty((N, 128), device="cuda")
    with pytest.raises(bsr.BsrError) as e:   # K mismatch
        bsr.bsr_spmm_batch([h1, h2], X, None, [Y1, Y2], N)
    assert e.value.status == 2   # BSR_ERR_SHAPE
    with pytest.raises(bsr.BsrError):        # the same handle twice
        bsr.bsr_spmm_batch([h1, h1], X, None, [Y1, Y2], N)
    with pytest.raises(bsr.BsrError):        # an output overlapping X
        bsr.bsr_spmm_batch([h1], X, None, [X.view(-1)[: N * 128].view(N, 128)], N)
    with pytest.raises(bsr.BsrError):        # two outputs overlapping each other
        w3 = _weight(1804, 128, 256, 8, 1, "f32", 0.2)
        h3, = _handles([w3], N)
        bsr.bsr_spmm_batch([h1, h3], X, None, [Y1, Y1], N)
    Xh = torch.from_numpy(synth.activations(1803, N, 256, "f32"))
    with pytest.raises(bsr.BsrError):        # host buffers are not accepted
        bsr.bsr_spmm_batch([h1], Xh, None, [Y1], N)
    bsr.bsr_spmm_batch([], X, None, [], N)   # empty batch: no-op
    bsr.bsr_spmm_batch([h1], X, None, [Y1], 0)
