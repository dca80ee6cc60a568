"""Chains of products on one stream with no synchronisation between calls.

The kernels are launched with programmatic stream serialisation: each one
may start its prologue while the previous kernel of the stream is still
running, and must wait for it before it reads X or the bias, or writes Y or
its workspace. A chain where each call's X is the previous call's Y, and a
call that overwrites an earlier call's X, would read stale or clobbered data
if a kernel touched those buffers too early. Every output is checked against
the oracle applied to the device's own input for that call (Section 2.2's
product, element by element within the fp32 / bf16 tolerance).
"""
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


def _layer(seed, M, K, R, C, dtype, density, long_rows=()):
    MB, KB = M // R, K // C
    if long_rows:
        cnt = np.full(MB, max(1, int(KB * density)), dtype=np.int64)
        cnt[list(long_rows)] = KB
        mask = synth.mask_from_row_counts(seed, cnt, KB)
    else:
        mask = synth.uniform_block_mask(seed, MB, KB, max(1, int(round(MB * KB * density))))
    return synth.make_weight("c", seed, M, K, R, C, dtype, 0, mask=mask)


def _run_chain(layers, N, dtype, seed, overwrite_input_last=False):
    """layers: weights whose K matches the previous M. Returns the host copies
    of every call's input and output, taken after one synchronisation."""
    bsr = _bsr()
    handles = []
    for w in layers:
        h = bsr.bsr_create(*build_on_gpu(w.W, w.R, w.C), w.R, w.C, w.M, w.K)
        h.reserve(N)
        handles.append(h)
    X0 = synth.activations(seed, N, layers[0].K, dtype)
    bufs = [to_dev(X0)]
    biases = [to_dev(w.bias) for w in layers]
    torch.cuda.synchronize()
    s = torch.cuda.current_stream()
    for i, (h, w) in enumerate(zip(handles, layers)):
        last = i == len(layers) - 1
        if last and overwrite_input_last:
            assert bufs[0].shape == (N, w.M)
            Y = bufs[0]   # the chain's first input, read by the first call, written by the last
        else:
            Y = torch.empty((N, w.M), device="cuda", dtype=bufs[0].dtype)
        bsr.bsr_spmm(h, bufs[i], biases[i], Y, N, s)
        bufs.append(Y)
    torch.cuda.synchronize()
    for h in handles:
        assert h.check_device_status() == 0
    outs = [to_host(b) for b in bufs[1:]]
    ins = [X0] + outs[:-1]
    return handles, ins, outs


def _check(layers, ins, outs):
    for w, X, Y in zip(layers, ins, outs):
        check_product(Y, oracle.bsr_from_dense(w.W, w.R, w.C), X, w.bias, w.M)


def test_fp32_chain_through_every_kernel_kind():
    """X -> 1x1 (one-row xstage) -> 32x32 (tensor cores, 3xTF32) -> 32x1
    (xstage, split items) -> 16x1 with long rows (xstage + split-row reduce)
    -> 3x2 (generic kernel) -> 2x1 on K = 255 (generic) written over X."""
    N = 200
    layers = [
        _layer(1201, 512, 256, 1, 1, "f32", 0.2),
        _layer(1202, 256, 512, 32, 32, "f32", 0.3),
        _layer(1203, 512, 256, 32, 1, "f32", 0.2),
        _layer(1204, 256, 512, 16, 1, "f32", 0.05, long_rows=(1, 7)),
        _layer(1205, 255, 256, 3, 2, "f32", 0.2),
        _layer(1206, 256, 255, 2, 1, "f32", 0.2),
    ]
    handles, ins, outs = _run_chain(layers, N, "f32", 1207, overwrite_input_last=True)
    kinds = [h.schedule()["variant"] for h in handles]
    assert kinds[0] == "xstage" and kinds[1] == "tcgen05" and kinds[2] == "xstage"
    assert kinds[3] == "xstage" and handles[3].schedule()["split_rows"] >= 1
    assert kinds[4] == "generic" and kinds[5] == "generic"
    _check(layers, ins, outs)


def test_bf16_chain_tensor_core_and_simt():
    """bf16: 16x16 (tensor cores) -> sparse 1x1 (xstage) -> 32x32 (tensor
    cores) -> dense 1x1 (re-blocked into 16-row tiles for the tensor cores) ->
    32x1, each call's X the previous call's Y."""
    N = 333
    layers = [
        _layer(1301, 512, 256, 16, 16, "bf16", 0.3),
        _layer(1302, 256, 512, 1, 1, "bf16", 0.06),
        _layer(1303, 512, 256, 32, 32, "bf16", 0.3),
        _layer(1306, 256, 512, 1, 1, "bf16", 0.3),
        _layer(1304, 512, 256, 32, 1, "bf16", 0.2),
    ]
    handles, ins, outs = _run_chain(layers, N, "bf16", 1305)
    kinds = [h.schedule()["variant"] for h in handles]
    assert kinds[:4] == ["tcgen05", "xstage", "tcgen05", "tcgen05"]
    assert handles[3].schedule()["exec_R"] == 16
    _check(layers, ins, outs)


def test_repeated_calls_overwrite_their_own_input():
    """One handle applied in place of its input's buffer pair, back and forth
    (square weight): call k reads buffer k % 2 and writes the other, ten
    calls queued with no synchronisation."""
    bsr = _bsr()
    N, M = 130, 256
    w = _layer(1401, M, M, 4, 4, "f32", 0.25)
    h = bsr.bsr_create(*build_on_gpu(w.W, 4, 4), 4, 4, M, M)
    h.reserve(N)
    X0 = synth.activations(1402, N, M, "f32")
    a, b = to_dev(X0), torch.empty((N, M), device="cuda")
    bias = to_dev(w.bias)
    torch.cuda.synchronize()
    for k in range(10):
        src, dst = (a, b) if k % 2 == 0 else (b, a)
        bsr.bsr_spmm(h, src, bias, dst, N)
    torch.cuda.synchronize()
    assert h.check_device_status() == 0
    # call 9 read b (call 8's output, not written since) and wrote a
    got = to_host(a)
    check_product(got, oracle.bsr_from_dense(w.W, 4, 4), to_host(b), w.bias, M)
    again = torch.empty((N, M), device="cuda")
    bsr.bsr_spmm(h, b, bias, again, N)
    torch.cuda.synchronize()
    assert np.array_equal(got, to_host(again)), "the queued call differs from the same call run alone"
