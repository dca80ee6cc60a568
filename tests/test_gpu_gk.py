"""The gathered-K tensor-core kernel (gk): each block row's kept columns of X
gathered into the MMA's A operand in tensor memory, fp32 as 3xTF32, bf16
directly. By default it takes the calls (of 512 or more tokens) of block
shapes that no specialised kernel runs, fp32 blocks of 64 or more rows; with
BSR_GK=1 it takes every shape it supports, which a subprocess sweep checks.
Every output element is compared with the oracle at the fp32 / bf16
tolerance."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import build_on_gpu, check_product, to_dev, to_host

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bsr():
    import paper_2106_08846_gb300 as bsr
    return bsr


def _weight(seed, M, K, R, C, dtype, density, dense=(), empty=()):
    MB, KB = M // R, K // C
    cnt = np.full(MB, max(1, int(round(KB * density))), dtype=np.int64)
    cnt[list(dense)] = KB
    cnt[list(empty)] = 0
    return synth.make_weight("gk", seed, M, K, R, C, dtype, 0, mask=synth.mask_from_row_counts(seed, cnt, KB))


@pytest.mark.parametrize("R,C", [(64, 1), (64, 4), (64, 8), (128, 2), (128, 8)])
def test_gk_runs_the_shapes_of_the_generic_kernel(R, C):
    # fp32 blocks of 64 and 128 rows: the generic kernel's shapes; 1000 tokens
    # go to gk (ragged last tile), 300 to the generic kernel
    bsr = _bsr()
    w = _weight(4100 + R + C, 512, 768, R, C, "f32", 0.15, dense=(1,), empty=(2,))
    h = bsr.bsr_create(*build_on_gpu(w.W, R, C), R, C, w.M, w.K)
    sc = h.schedule()
    assert sc["variant"] == "generic" and sc["gk_task_sizes"] != "none"
    ref = oracle.bsr_from_dense(w.W, R, C)
    for N in (1000, 300):
        X = synth.activations(4200 + N, N, w.K, "f32")
        Y = h.spmm(to_dev(X), to_dev(w.bias))
        torch.cuda.synchronize()
        assert h.check_device_status() == 0
        check_product(to_host(Y), ref, X, w.bias, w.M)


@pytest.mark.parametrize("env", [{}, {"BSR_GK_G": "1"}, {"BSR_GK_G": "2"}])
def test_gk_forced_on_every_supported_shape(env):
    # every task size the kernel chooses, one-row tasks (many tasks per CTA
    # range: the double-buffered records) and two-row tasks
    e = dict(os.environ, BSR_GK="1", **env)
    r = subprocess.run([sys.executable, "-m", "tests.gk_forced_check"], cwd=ROOT, env=e, capture_output=True,
                       text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert r.stdout.count(": ok") == r.stdout.count("\n")


def test_gk_bounded_wait_times_out_and_reports(monkeypatch):
    """An X chunk that is never loaded: the waits give up after the bound
    (2 ms), the kernel records BSR_ERR_TIMEOUT, drains its copies, waits for
    its MMAs, frees the tensor memory and returns; the context stays usable."""
    bsr = _bsr()
    from paper_2106_08846_gb300 import bsrlib as b
    w = _weight(4300, 512, 768, 64, 4, "f32", 0.15)
    gpu = build_on_gpu(w.W, 64, 4)
    monkeypatch.setenv("BSR_WAIT_LIMIT_NS", "2000000")
    monkeypatch.setenv("BSR_TEST_STALL_CHUNK", "1")
    h = bsr.bsr_create(*gpu, 64, 4, w.M, w.K)
    monkeypatch.delenv("BSR_WAIT_LIMIT_NS")
    monkeypatch.delenv("BSR_TEST_STALL_CHUNK")
    X = synth.activations(4301, 1000, w.K, "f32")
    h.spmm(to_dev(X), to_dev(w.bias))
    assert h.check_device_status() == b.BSR_ERR_TIMEOUT
    assert h.check_device_status() == b.BSR_OK
    h2 = bsr.bsr_create(*gpu, 64, 4, w.M, w.K)
    Y = to_host(h2.spmm(to_dev(X), to_dev(w.bias)))
    assert h2.check_device_status() == b.BSR_OK
    check_product(Y, oracle.bsr_from_dense(w.W, 64, 4), X, w.bias, w.M)


def test_gk_chain_without_synchronisation():
    """X -> 64x4 (gk) -> 32x1 (xstage) -> 128x2 (gk) written over X, queued
    with no synchronisation (programmatic launches)."""
    bsr = _bsr()
    N = 700
    layers = [_weight(4401, 512, 384, 64, 4, "f32", 0.2), _weight(4402, 384, 512, 32, 1, "f32", 0.15),
              _weight(4403, 384, 384, 128, 2, "f32", 0.2)]
    handles = [bsr.bsr_create(*build_on_gpu(w.W, w.R, w.C), w.R, w.C, w.M, w.K) for w in layers]
    for h in handles:
        h.reserve(N)
    X0 = synth.activations(4404, N, 384, "f32")
    x0 = to_dev(X0)
    outs = [torch.empty((N, 512), device="cuda"), torch.empty((N, 384), device="cuda"), x0]
    src = x0
    torch.cuda.synchronize()
    for h, w, Y in zip(handles, layers, outs):
        bsr.bsr_spmm(h, src, to_dev(w.bias), Y, N, torch.cuda.current_stream())
        src = Y
    torch.cuda.synchronize()
    ins = [X0, to_host(outs[0]), to_host(outs[1])]
    for h, w, X, Y in zip(handles, layers, ins, outs):
        assert h.check_device_status() == 0
        check_product(to_host(Y), oracle.bsr_from_dense(w.W, w.R, w.C), X, w.bias, w.M)
