"""The persistent SIMT kernel for tall blocks (16 or 32 rows, one column or
16 / 32 columns) that takes bsr_spmm calls with enough tokens to give every
SM at least one unit of work. Each case checks that the call runs on it (the
same rule the library applies) and compares every output element with the
oracle at the fp32 / bf16 tolerance: shapes and dtypes, ragged token tails,
tasks that change inside one CTA's range, split and empty rows, the 128-token
configuration, a chain of calls with no synchronisation, and a bounded wait
that runs out."""
import math

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


def xrow_config(h, N):
    """The configuration the library picks for N tokens (-1: the xstage kernel)."""
    sc = h.schedule()
    if sc["variant"] != "xstage":
        return -1
    tasks = [int(t) for t in str(sc["xrow_tasks"]).split(",")]
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for s, t in enumerate(tasks):
        if t and t * math.ceil(N / (64 << s)) >= sms:
            return s
    return -1


def _create(w, monkeypatch=None, force_simt=False):
    bsr = _bsr()
    if force_simt:
        monkeypatch.setenv("BSR_FORCE_VARIANT", "xstage")
    h = bsr.bsr_create(*build_on_gpu(w.W, w.R, w.C), w.R, w.C, w.M, w.K)
    if force_simt:
        monkeypatch.delenv("BSR_FORCE_VARIANT")
    return h


def _check_call(h, w, N, seed, bias=True):
    X = synth.activations(seed, N, w.K, w.dtype)
    b = to_dev(w.bias) if bias else None
    Y = h.spmm(to_dev(X), b)
    torch.cuda.synchronize()
    assert h.check_device_status() == 0
    check_product(to_host(Y), oracle.bsr_from_dense(w.W, w.R, w.C), X, w.bias if bias else None, w.M)


def _uniform(seed, M, K, R, C, dtype, density):
    MB, KB = M // R, K // C
    mask = synth.uniform_block_mask(seed, MB, KB, max(1, int(round(MB * KB * density))))
    return synth.make_weight("xr", seed, M, K, R, C, dtype, 0, mask=mask)


@pytest.mark.parametrize("R,C,density", [(32, 1, 0.12), (16, 1, 0.12), (16, 16, 0.25), (32, 16, 0.25),
                                         (16, 32, 0.25), (32, 32, 0.25)])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_xrow_parity(monkeypatch, R, C, density, dtype):
    # 5000 tokens: 79 tiles of 64 (the last holds 8), several tasks, so CTA
    # ranges cross task boundaries; shapes the tensor cores would take
    # (bf16, and fp32 blocks of 32 rows and 16 or more columns) forced onto
    # the SIMT kernels
    w = _uniform(3000 + R + C, 384, 768, R, C, dtype, density)
    h = _create(w, monkeypatch, force_simt=True)
    N = 5000
    assert xrow_config(h, N) >= 0   # (wide blocks may need the 128-token configuration)
    _check_call(h, w, N, 3001 + R)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_xrow_without_bias(monkeypatch, dtype):
    w = _uniform(3100, 384, 512, 32, 1, dtype, 0.1)
    h = _create(w, monkeypatch, force_simt=dtype == "bf16")
    assert xrow_config(h, 5000) == 0
    _check_call(h, w, 5000, 3101, bias=False)


@pytest.mark.parametrize("R,C,K", [(32, 1, 512), (16, 16, 1024)])
def test_xrow_split_and_empty_rows(R, C, K):
    # dense rows split into pieces (fp32 partials and the reduce pass), empty
    # rows (no item: the reduce pass writes the bias), short rows elsewhere
    M = 512
    MB, KB = M // R, K // C
    cnt = np.full(MB, max(1, KB // 10), dtype=np.int64)
    cnt[[3, MB // 2]] = KB
    cnt[[5, MB - 1]] = 0
    w = synth.make_weight("xs", 3200 + R, M, K, R, C, "f32", 0, mask=synth.mask_from_row_counts(3200 + R, cnt, KB))
    h = _create(w)
    sc = h.schedule()
    assert sc["split_rows"] >= 2 and sc["empty_rows"] >= 2
    N = 4000
    assert xrow_config(h, N) >= 0
    _check_call(h, w, N, 3201)


def test_xrow_128_token_configuration():
    # rows of about 205 blocks: six items of a 64-token task do not fit shared
    # memory, three of a 128-token task do (4900 tokens: the last tile holds 36)
    w = _uniform(3300, 384, 2048, 32, 1, "f32", 0.1)
    h = _create(w)
    tasks = [int(t) for t in str(h.schedule()["xrow_tasks"]).split(",")]
    assert tasks[0] == 0 and tasks[1] > 0
    N = 4900
    assert xrow_config(h, N) == 1
    _check_call(h, w, N, 3301)


def test_xrow_chain_without_synchronisation():
    """X -> 32x1 -> 16x16 -> 32x1 written over X, queued with no
    synchronisation (programmatic launches: each kernel may start while the
    previous one runs, and waits before it touches X, the bias or Y)."""
    bsr = _bsr()
    N = 5000
    layers = [_uniform(3401, 512, 384, 32, 1, "f32", 0.15), _uniform(3402, 384, 512, 16, 16, "f32", 0.25),
              _uniform(3403, 384, 384, 32, 1, "f32", 0.15)]
    handles = [_create(w) for w in layers]
    for h in handles:
        h.reserve(N)
        assert xrow_config(h, N) >= 0
    X0 = synth.activations(3404, N, 384, "f32")
    bufs = [to_dev(X0)]
    s = torch.cuda.current_stream()
    torch.cuda.synchronize()
    outs = [torch.empty((N, 512), device="cuda"), torch.empty((N, 384), device="cuda"), bufs[0]]
    for h, w, Y in zip(handles, layers, outs):
        bsr.bsr_spmm(h, bufs[-1], to_dev(w.bias), Y, N, s)
        bufs.append(Y)
    torch.cuda.synchronize()
    ins = [X0, to_host(outs[0]), to_host(outs[1])]
    for h, w, X, Y in zip(handles, layers, ins, outs):
        assert h.check_device_status() == 0
        check_product(to_host(Y), oracle.bsr_from_dense(w.W, w.R, w.C), X, w.bias, w.M)


def test_xrow_bounded_wait_times_out_and_reports(monkeypatch):
    """An X chunk that is never loaded: the consumers' wait gives up after the
    bound (2 ms), the kernel records BSR_ERR_TIMEOUT, drains its copies and
    returns; the context stays usable and a normal handle computes correctly."""
    bsr = _bsr()
    from paper_2106_08846_gb300 import bsrlib as b
    w = _uniform(3500, 384, 768, 32, 1, "f32", 0.12)
    gpu = build_on_gpu(w.W, 32, 1)
    monkeypatch.setenv("BSR_WAIT_LIMIT_NS", "2000000")
    monkeypatch.setenv("BSR_TEST_STALL_CHUNK", "1")
    h = bsr.bsr_create(*gpu, 32, 1, w.M, w.K)
    monkeypatch.delenv("BSR_WAIT_LIMIT_NS")
    monkeypatch.delenv("BSR_TEST_STALL_CHUNK")
    N = 5000
    assert xrow_config(h, N) == 0
    X = synth.activations(3501, N, w.K, "f32")
    h.spmm(to_dev(X), to_dev(w.bias))
    assert h.check_device_status() == b.BSR_ERR_TIMEOUT
    assert h.check_device_status() == b.BSR_OK
    h2 = bsr.bsr_create(*gpu, 32, 1, w.M, w.K)
    Y = to_host(h2.spmm(to_dev(X), to_dev(w.bias)))
    assert h2.check_device_status() == b.BSR_OK
    check_product(Y, oracle.bsr_from_dense(w.W, 32, 1), X, w.bias, w.M)
