"""GPU path vs the CPU oracle through the C ABI: the builder bit for bit, the
product within |dY| <= tol * (sum |x||w| + |b|) (tol 1e-5 fp32, 1e-2 bf16),
at sizes spanning several tiles with ragged tails, plus edge cases and the
documented error statuses."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import (assert_structure_equal, build_on_gpu, check_product, to_dev, to_host)

pytestmark = pytest.mark.gpu

SHAPES = [(1, 1), (4, 4), (8, 1), (16, 1), (32, 1), (1, 32), (16, 16), (32, 32), (2, 3), (64, 64)]


def _bsr():
    import paper_2106_08846_gb300 as bsr
    return bsr


def _weight(M, K, R, C, dtype, density, seed):
    MB, KB = M // R, K // C
    mask = synth.uniform_block_mask(seed, MB, KB, int(round(MB * KB * density)))
    return synth.make_weight("t", seed, M, K, R, C, dtype, 0, mask=mask)


def _run(w, X, bias=True, dev_bias=None):
    bsr = _bsr()
    gpu = build_on_gpu(w.W, w.R, w.C)
    h = bsr.bsr_create(*gpu, w.R, w.C, w.M, w.K)
    b = to_dev(w.bias) if bias else None
    Y = h.spmm(to_dev(X), b)
    torch.cuda.synchronize()
    assert h.check_device_status() == 0
    return h, gpu, to_host(Y)


# ---------------------------------------------------------------- builder

@pytest.mark.parametrize("R,C", SHAPES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_builder_bit_exact(R, C, dtype):
    M, K = 192, 320
    if M % R or K % C:
        M, K = R * 6, C * 10
    w = _weight(M, K, R, C, dtype, 0.3, 1000 + R * 10 + C)
    assert_structure_equal(build_on_gpu(w.W, R, C), oracle.bsr_from_dense(w.W, R, C))


@pytest.mark.parametrize("thr", [0.0, 0.01, 0.03, 1e30])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_builder_thresholds(thr, dtype):
    w = _weight(256, 256, 16, 16, dtype, 0.5, 77)
    assert_structure_equal(build_on_gpu(w.W, 4, 4, thr), oracle.bsr_from_dense(w.W, 4, 4, thr))


def test_builder_special_values():
    W = np.zeros((8, 32), dtype=np.float32)
    W[0, 0] = np.nan
    W[1, 4] = -0.0
    W[2, 8] = 1e-45
    W[3, 12] = 0.25
    W[4, 16] = -0.2500001
    W[5, 20] = np.inf
    W[6, 24] = -np.inf
    for thr in (0.0, 0.25):
        ref = oracle.bsr_from_dense(W, 2, 4, thr)
        assert_structure_equal(build_on_gpu(W, 2, 4, thr), ref)


def test_builder_empty_and_full():
    for W in (np.zeros((64, 96), np.float32), np.ones((64, 96), np.float32)):
        assert_structure_equal(build_on_gpu(W, 8, 8), oracle.bsr_from_dense(W, 8, 8))


def test_builder_query_and_capacity():
    import ctypes
    bsr = _bsr()
    lib = bsr.load()
    w = _weight(128, 128, 8, 1, "f32", 0.2, 5)
    Wd = to_dev(w.W)
    indptr = torch.empty(17, dtype=torch.int32, device="cuda")
    n = ctypes.c_int64(-1)
    st = lib.bsr_from_dense(ctypes.c_void_p(Wd.data_ptr()), 128, 128, 8, 1, 0.0, 0,
                            ctypes.c_void_p(indptr.data_ptr()), None, None, 0, ctypes.byref(n), None)
    assert st == 0 and n.value == w.nnzb
    idx = torch.full((n.value - 1,), -7, dtype=torch.int32, device="cuda")
    data = torch.empty((n.value - 1, 8, 1), dtype=torch.float32, device="cuda")
    st = lib.bsr_from_dense(ctypes.c_void_p(Wd.data_ptr()), 128, 128, 8, 1, 0.0, 0,
                            ctypes.c_void_p(indptr.data_ptr()), ctypes.c_void_p(idx.data_ptr()),
                            ctypes.c_void_p(data.data_ptr()), n.value - 1, ctypes.byref(n), None)
    assert st == bsr.bsrlib.BSR_ERR_CAPACITY and n.value == w.nnzb
    assert (idx == -7).all()
    assert np.array_equal(to_host(indptr), oracle.bsr_from_dense(w.W, 8, 1)[0])


# ---------------------------------------------------------------- product

@pytest.mark.parametrize("R,C", SHAPES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N", [1, 77, 300])
def test_spmm_parity(R, C, dtype, N):
    M, K = 256, 384
    if M % R or K % C:
        M, K = R * 40, C * 60
    w = _weight(M, K, R, C, dtype, 0.2, 2000 + R * 10 + C)
    X = synth.activations(3000 + N, N, K, dtype)
    _, _, Y = _run(w, X)
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


@pytest.mark.parametrize("R,C", [(32, 1), (16, 16), (1, 1), (8, 1)])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_spmm_uneven_rows_split(R, C, dtype):
    """A few fully dense block rows among short and empty ones: the long rows
    are split into pieces and summed by the reduce pass."""
    M, K = 512, 2048
    MB, KB = M // R, K // C
    seed = 4000 + R + C
    cnt = np.zeros(MB, dtype=np.int64)
    cnt[1::2] = 2
    cnt[[3, MB // 2, MB - 2]] = KB
    w = synth.make_weight("z", seed, M, K, R, C, dtype, 0, mask=synth.mask_from_row_counts(seed, cnt, KB))
    X = synth.activations(seed, 150, K, dtype)
    h, _, Y = _run(w, X)
    sched = h.schedule()
    assert sched["empty_rows"] == int((cnt == 0).sum())
    if sched["exec_C"] == C:   # (narrow bf16 blocks re-blocked into 64-column tiles need no split here)
        assert sched["split_rows"] == 3
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


@pytest.mark.parametrize("R,C", [(32, 1), (16, 16)])
def test_spmm_zipf_rows(R, C):
    M, K = 512, 1024
    MB, KB = M // R, K // C
    seed = 4100 + R + C
    cnt = synth.zipf_row_counts(seed, MB, KB, MB * KB // 20)
    w = synth.make_weight("z", seed, M, K, R, C, "bf16", 95, mask=synth.mask_from_row_counts(seed, cnt, KB))
    X = synth.activations(seed, 150, K, "bf16")
    _, _, Y = _run(w, X)
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_spmm_no_blocks_gives_bias_exactly(dtype):
    bsr = _bsr()
    M, K, N = 128, 64, 33
    W = np.zeros((M, K), dtype=np.float32 if dtype == "f32" else np.uint16)
    b = synth.normal(1, synth.STREAM_BIAS, M, 0.02)
    X = synth.activations(2, N, K, dtype)
    gpu = build_on_gpu(W, 16, 16)
    assert to_host(gpu[0]).sum() == 0 and gpu[1].numel() == 0
    h = bsr.bsr_create(*gpu, 16, 16, M, K)
    Y = to_host(h.spmm(to_dev(X), to_dev(b)))
    want = np.broadcast_to(b, (N, M)) if dtype == "f32" else np.broadcast_to(oracle.round_bf16(b.astype(np.float64)), (N, M))
    assert Y.tobytes() == np.ascontiguousarray(want).tobytes()
    Y0 = to_host(h.spmm(to_dev(X), None))
    assert not Y0.any()


def test_spmm_without_bias_and_n_zero():
    bsr = _bsr()
    w = _weight(128, 256, 32, 1, "f32", 0.1, 9)
    X = synth.activations(10, 40, 256, "f32")
    h, gpu, Y = _run(w, X, bias=False)
    check_product(Y, oracle.bsr_from_dense(w.W, 32, 1), X, None, 128)
    Yd = torch.full((5, 128), 3.0, device="cuda")
    bsr.bsr_spmm(h, to_dev(X), None, Yd, 0)
    torch.cuda.synchronize()
    assert (Yd == 3.0).all()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_spmm_host_buffers_match_device(dtype):
    w = _weight(256, 512, 16, 16, dtype, 0.15, 12)
    X = synth.activations(13, 99, 512, dtype)
    h, _, Y = _run(w, X)
    Xh = to_dev(X, "cpu").pin_memory()
    Yh = torch.empty((99, 256), dtype=Xh.dtype).pin_memory()
    bias = to_dev(w.bias)
    _bsr().bsr_spmm(h, Xh, bias, Yh, 99)
    torch.cuda.synchronize()
    assert to_host(Yh).tobytes() == Y.tobytes()


def test_spmm_empty_rows_mixed():
    M, K, R, C = 256, 256, 8, 1
    mask = synth.uniform_block_mask(14, M // R, K // C, 600)
    mask[::3] = False
    w = synth.make_weight("e", 14, M, K, R, C, "f32", 0, mask=mask)
    X = synth.activations(15, 65, K, "f32")
    _, _, Y = _run(w, X)
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


def test_schedule_cache_reuses_identical_structure():
    bsr = _bsr()
    w = _weight(256, 256, 32, 1, "f32", 0.2, 16)
    gpu = build_on_gpu(w.W, 32, 1)
    h1 = bsr.bsr_create(*gpu, 32, 1, 256, 256)
    h2 = bsr.bsr_create(*gpu, 32, 1, 256, 256)
    s1, s2 = h1.schedule(), h2.schedule()
    assert s2["cache_hit"] == 1 and s2["structure_hash"] == s1["structure_hash"]
    assert s2["schedule_reuses"] >= 1
    w2 = _weight(256, 256, 32, 1, "f32", 0.2, 17)
    h3 = bsr.bsr_create(*build_on_gpu(w2.W, 32, 1), 32, 1, 256, 256)
    assert h3.schedule()["cache_hit"] == 0


def test_reserve_then_spmm():
    w = _weight(128, 128, 16, 16, "bf16", 0.3, 18)
    bsr = _bsr()
    h = bsr.bsr_create(*build_on_gpu(w.W, 16, 16), 16, 16, 128, 128)
    h.reserve(512)
    X = synth.activations(19, 512, 128, "bf16")
    Y = to_host(h.spmm(to_dev(X), to_dev(w.bias)))
    check_product(Y, oracle.bsr_from_dense(w.W, 16, 16), X, w.bias, 128)


# ---------------------------------------------------------------- errors

def test_error_statuses():
    bsr = _bsr()
    from paper_2106_08846_gb300 import bsrlib as b
    import ctypes
    lib = bsr.load()
    w = _weight(128, 128, 8, 1, "f32", 0.2, 20)
    gpu = build_on_gpu(w.W, 8, 1)
    h = bsr.bsr_create(*gpu, 8, 1, 128, 128)
    X = torch.zeros((10, 128), device="cuda")
    Y = torch.zeros((10, 128), device="cuda")
    P = ctypes.c_void_p
    # misaligned X
    st = lib.bsr_spmm(h.ptr, P(X.data_ptr() + 4), None, P(Y.data_ptr()), 9, None)
    assert st == b.BSR_ERR_ALIGNMENT
    # X and Y overlap
    st = lib.bsr_spmm(h.ptr, P(X.data_ptr()), None, P(X.data_ptr() + 64), 4, None)
    assert st == b.BSR_ERR_INVALID_ARG
    # host X with device Y
    Xh = torch.zeros((10, 128)).pin_memory()
    st = lib.bsr_spmm(h.ptr, P(Xh.data_ptr()), None, P(Y.data_ptr()), 10, None)
    assert st == b.BSR_ERR_INVALID_ARG
    # bad structures
    indptr, indices, data = (t.clone() for t in gpu)
    out = P()

    def create(ip, ix):
        return lib.bsr_create(P(ip.data_ptr()), P(ix.data_ptr()), P(data.data_ptr()), 8, 1, 128, 128, 0,
                              ctypes.byref(out))
    bad = indices.clone()
    row0 = int(indptr[1])
    if row0 >= 2:
        bad[0], bad[1] = indices[1], indices[0]
        assert create(indptr, bad) == b.BSR_ERR_STRUCTURE
    bad = indices.clone()
    bad[-1] = 128
    assert create(indptr, bad) == b.BSR_ERR_STRUCTURE
    bad_ip = indptr.clone()
    bad_ip[0] = 1
    assert create(bad_ip, indices) == b.BSR_ERR_STRUCTURE
    bad_ip = indptr.clone()
    bad_ip[3] = bad_ip[2] - 1
    assert create(bad_ip, indices) == b.BSR_ERR_STRUCTURE
    assert create(indptr, indices) == b.BSR_OK
    lib.bsr_destroy(out)
    # host arrays are not accepted by bsr_create
    assert lib.bsr_create(P(indptr.cpu().data_ptr()), P(indices.data_ptr()), P(data.data_ptr()), 8, 1, 128,
                          128, 0, ctypes.byref(out)) == b.BSR_ERR_INVALID_ARG
    assert h.check_device_status() == b.BSR_OK


@pytest.mark.parametrize("R,C,dtype,variant,N", [(32, 1, "f32", "xstage", 5000), (32, 1, "f32", "xstage", 128),
                                                 (16, 16, "bf16", "tcgen05", 128), (32, 32, "f32", "tcgen05", 128)])
def test_bounded_wait_times_out_and_reports(monkeypatch, R, C, dtype, variant, N):
    """An X chunk that is never loaded: every wait on it gives up after the
    bound (2 ms here), the kernel records BSR_ERR_TIMEOUT, releases what it
    holds and returns; the context stays usable and a normal handle still
    computes correctly. The SIMT kernel runs once with many token tiles per
    task (the stalled chunk's waits end in every CTA at once) and once with
    two."""
    bsr = _bsr()
    from paper_2106_08846_gb300 import bsrlib as b
    w = _weight(256, 512, R, C, dtype, 0.2, 21)
    gpu = build_on_gpu(w.W, R, C)
    monkeypatch.setenv("BSR_WAIT_LIMIT_NS", "2000000")
    monkeypatch.setenv("BSR_TEST_STALL_CHUNK", "1")
    h = bsr.bsr_create(*gpu, R, C, 256, 512)
    monkeypatch.delenv("BSR_WAIT_LIMIT_NS")
    monkeypatch.delenv("BSR_TEST_STALL_CHUNK")
    assert h.schedule()["variant"] == variant
    X = synth.activations(22, N, 512, dtype)
    h.spmm(to_dev(X), to_dev(w.bias))
    assert h.check_device_status() == b.BSR_ERR_TIMEOUT
    assert h.check_device_status() == b.BSR_OK          # cleared after reading
    h2 = bsr.bsr_create(*gpu, R, C, 256, 512)
    Y = to_host(h2.spmm(to_dev(X), to_dev(w.bias)))
    assert h2.check_device_status() == b.BSR_OK
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, 256)


@pytest.mark.parametrize("R,C", [(16, 16), (32, 32), (64, 64), (16, 32), (32, 16)])
def test_tensor_core_path_is_used_for_bf16_square_blocks(R, C):
    w = _weight(256, 512, R, C, "bf16", 0.25, 30 + R + C)
    X = synth.activations(31, 200, 512, "bf16")
    h, _, Y = _run(w, X)
    assert h.schedule()["variant"] == "tcgen05"
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, 256)


@pytest.mark.parametrize("R,C", [(32, 32), (32, 16), (64, 16), (64, 32)])
def test_tensor_core_path_is_used_for_fp32_square_blocks(R, C):
    """fp32 blocks with both sides multiples of 16 run on the tensor cores as
    three tf32 products (high x high + high x low + low x high) and must meet
    the fp32 tolerance."""
    w = _weight(256, 512, R, C, "f32", 0.25, 40 + R + C)
    X = synth.activations(41, 200, 512, "f32")
    h, _, Y = _run(w, X)
    assert h.schedule()["variant"] == "tcgen05"
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, 256)


def test_fp32_tensor_core_path_handles_large_magnitudes_and_tails():
    """3xTF32 keeps fp32 accuracy across magnitudes: inputs scaled over a wide
    range, a ragged token tail and K not a multiple of the 32-column stage."""
    R, C = 32, 16
    w = _weight(128, 16 * 21, R, C, "f32", 0.4, 77)
    X = synth.activations(78, 131, 16 * 21, "f32") * np.float32(3.0e3)
    X[::7] *= np.float32(1e-3)
    h, _, Y = _run(w, X)
    assert h.schedule()["variant"] == "tcgen05"
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, w.M)


@pytest.mark.parametrize("R,C", [(32, 1), (16, 1), (16, 4), (64, 2)])
def test_narrow_bf16_blocks_run_as_tensor_core_tiles(R, C):
    """Dense enough narrow bf16 blocks are re-blocked into zero-filled R x 64
    tiles for the tensor cores; the product matches the oracle on the
    original blocks, with a ragged token tail and a partial last tile."""
    M, K = 256, 64 * 7 + 16 * C
    w = _weight(M, K, R, C, "bf16", 0.5, 50 + R + C)
    X = synth.activations(51, 210, K, "bf16")
    h, _, Y = _run(w, X)
    s = h.schedule()
    assert s["variant"] == "tcgen05" and s["exec_C"] == 64
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


@pytest.mark.parametrize("R,C", [(1, 1), (1, 32), (4, 4), (8, 1), (2, 16), (8, 8)])
def test_small_bf16_blocks_run_as_16_row_tensor_core_tiles(R, C):
    """bf16 blocks of fewer than 16 rows, dense enough, stack 16 / R block rows
    into zero-filled 16 x 64 tiles for the tensor cores; the product matches
    the oracle on the original blocks (ragged tokens, a partial last tile,
    rows without blocks)."""
    M, K = 256, 64 * 5 + 32
    MB, KB = M // R, K // C
    cnt = np.full(MB, max(1, int(KB * 0.35)), dtype=np.int64)
    cnt[[3, MB // 2]] = 0   # rows without blocks (their tile rows still hold other rows' blocks)
    w = synth.make_weight("t", 70 + R + C, M, K, R, C, "bf16", 0,
                          mask=synth.mask_from_row_counts(70 + R + C, cnt, KB))
    X = synth.activations(71, 210, K, "bf16")
    h, _, Y = _run(w, X)
    s = h.schedule()
    assert s["variant"] == "tcgen05" and s["exec_R"] == 16 and s["exec_C"] == 64
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


@pytest.mark.parametrize("holes", [False, True])
def test_stacked_mmas_for_dense_tile_rows(holes):
    """Re-blocked 32x1 bf16 tiles where every tile row of a task has a tile in
    a chunk run as one MMA over all the task's rows (a stack: N = rows x 32).
    With holes, one tile row has no tile in chunk 2 and another starts in
    chunk 1, so some chunks mix stacked and per-item MMAs in one task; the
    product must match the oracle either way (many token tiles, ragged tail)."""
    R, C, M, K, N = 32, 1, 256, 512, 5000
    MB, KB = M // R, K // C
    mask = synth.uniform_block_mask(90, MB, KB, int(MB * KB * 0.3))
    if holes:
        mask[3, 128:192] = False
        mask[5, 0:64] = False
    w = synth.make_weight("s", 91, M, K, R, C, "bf16", 0, mask=mask)
    X = synth.activations(92, N, K, "bf16")
    h, _, Y = _run(w, X)
    s = h.schedule()
    assert s["variant"] == "tcgen05" and s["exec_R"] == 32 and s["exec_C"] == 64
    stacks = [int(v) for v in str(s["tc_stacked_chunks"]).split(",")]
    assert stacks[0] == 0 and all(v > 0 for v in stacks[1:4])   # G = 1 has nothing to stack; G = 2, 4, 8 do
    if holes:
        assert stacks[3] < K // 64   # the task of all eight rows cannot stack chunks 0, 1 and 2
    rows = np.concatenate([np.arange(0, 300), np.arange(N - 300, N)])
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M, rows=rows)


def test_stacked_mmas_for_32_column_bf16_blocks():
    """Native 32x32 bf16 blocks, every block kept, K = 96: the first 64-column
    chunk holds two blocks of every row (per-item MMAs), the second one block of
    every row at the same offset (a stack); ragged token tail."""
    R, C, M, K, N = 32, 32, 256, 96, 333
    mask = np.ones((M // R, K // C), dtype=bool)
    w = synth.make_weight("s32", 93, M, K, R, C, "bf16", 0, mask=mask)
    X = synth.activations(94, N, K, "bf16")
    h, _, Y = _run(w, X)
    s = h.schedule()
    assert s["variant"] == "tcgen05" and s["exec_C"] == 32
    stacks = [int(v) for v in str(s["tc_stacked_chunks"]).split(",")]
    assert stacks[0] == 0 and stacks[1] > 0
    check_product(Y, oracle.bsr_from_dense(w.W, R, C), X, w.bias, M)


@pytest.mark.parametrize("C", [16, 32])
def test_large_fp32_16_row_weights_run_3xtf32_small_ones_simt(C):
    """fp32 blocks of 16 rows: on a weight of 2^20 elements (1024 x 1024) the
    tensor cores take them as 3xTF32 (ragged tokens, split rows from a dense
    row, an empty row); on a 768 x 768 weight the SIMT kernel keeps them."""
    MB, KB = 1024 // 16, 1024 // C
    cnt = np.full(MB, KB // 10, dtype=np.int64)
    cnt[3], cnt[MB - 2] = KB, 0
    w = synth.make_weight("r16", 90 + C, 1024, 1024, 16, C, "f32", 0, mask=synth.mask_from_row_counts(90 + C, cnt, KB))
    X = synth.activations(91 + C, 333, 1024, "f32")
    h, _, Y = _run(w, X)
    assert h.schedule()["variant"] == "tcgen05"
    check_product(Y, oracle.bsr_from_dense(w.W, 16, C), X, w.bias, 1024)
    small = _weight(768, 768, 16, C, "f32", 0.2, 92)
    h2, _, Y2 = _run(small, synth.activations(93, 100, 768, "f32"))
    assert h2.schedule()["variant"] == "xstage"


def test_small_bf16_blocks_whose_rows_do_not_fill_tiles_stay_simt():
    """M not a multiple of 16 (4-row blocks, M = 260): no 16-row tiling, the
    SIMT kernel keeps the weight."""
    w = _weight(260, 256, 4, 4, "bf16", 0.4, 80)
    X = synth.activations(81, 100, 256, "bf16")
    h, _, Y = _run(w, X)
    assert h.schedule()["variant"] == "xstage"
    check_product(Y, oracle.bsr_from_dense(w.W, 4, 4), X, w.bias, 260)


def test_sparse_narrow_bf16_blocks_stay_simt():
    """Below about 5 kept columns per 64-column tile (1/12 fill) the padded
    tensor work is not worth it: the SIMT kernel keeps the weight."""
    w = _weight(256, 1024, 32, 1, "bf16", 0.02, 60)
    X = synth.activations(61, 64, 1024, "bf16")
    h, _, Y = _run(w, X)
    assert h.schedule()["variant"] == "xstage"
    check_product(Y, oracle.bsr_from_dense(w.W, 32, 1), X, w.bias, 256)


@pytest.mark.parametrize("R,C,dtype", [(32, 1, "f32"), (1, 1, "f32"), (16, 16, "bf16"), (32, 32, "f32")])
def test_spmm_captured_in_cuda_graph(R, C, dtype):
    """After bsr_reserve, bsr_spmm allocates nothing and synchronises nothing,
    so it can be captured in a CUDA graph: replays with new X match the oracle
    (the weight has split rows, so the split-row workspace is in the graph)."""
    M, K, N = 256, 512, 200
    MB, KB = M // R, K // C
    cnt = np.full(MB, max(1, KB // 10), dtype=np.int64)
    cnt[[1, MB // 2]] = KB   # long rows: split pieces and the reduce pass
    w = synth.make_weight("g", 900 + R + C, M, K, R, C, dtype, 0,
                          mask=synth.mask_from_row_counts(900 + R + C, cnt, KB))
    bsr = _bsr()
    h = bsr.bsr_create(*build_on_gpu(w.W, R, C), R, C, M, K)
    h.reserve(N)
    X0 = synth.activations(901, N, K, dtype)
    Xd = to_dev(X0)
    b = to_dev(w.bias)
    Y = torch.empty((N, M), device="cuda", dtype=Xd.dtype)
    bsr.bsr_spmm(h, Xd, b, Y, N)   # first call outside the capture (one-time kernel set-up)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        bsr.bsr_spmm(h, Xd, b, Y, N, torch.cuda.current_stream())
    ref = oracle.bsr_from_dense(w.W, R, C)
    for seed in (902, 903):
        X = synth.activations(seed, N, K, dtype)
        Xd.copy_(to_dev(X))
        g.replay()
        torch.cuda.synchronize()
        assert h.check_device_status() == 0
        check_product(to_host(Y), ref, X, w.bias, M)
