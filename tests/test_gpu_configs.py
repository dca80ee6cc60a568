"""The five benchmark workloads at full size, through the C ABI in the launch
configuration the benchmark uses. The oracle checks a sample of tokens one by
one (first, last and seeded random ones) for every weight; the builder is
checked bit for bit against the oracle for every weight."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import assert_structure_equal, build_on_gpu, check_product, to_dev, to_host

pytestmark = pytest.mark.gpu


def _sample_rows(N, k, seed):
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([[0, N - 1], rng.choice(N, size=min(k, N), replace=False)]))


def _check_workload(wl, sample=12):
    import paper_2106_08846_gb300 as bsr
    X = wl.make_X()
    Xd = to_dev(X)
    for i, w in enumerate(wl.weights):
        ref = oracle.bsr_from_dense(w.W, w.R, w.C)
        gpu = build_on_gpu(w.W, w.R, w.C)
        assert_structure_equal(gpu, ref)
        h = bsr.bsr_create(*gpu, w.R, w.C, w.M, w.K)
        Y = h.spmm(Xd, to_dev(w.bias))
        torch.cuda.synchronize()
        assert h.check_device_status() == 0
        Yh = to_host(Y)
        rows = _sample_rows(wl.N, sample, 17 + i)
        check_product(Yh, ref, X, w.bias, w.M, rows=rows)
        h.destroy()


def test_config1_bert_base_single_weight():
    wl = synth.config(1)
    _check_workload(wl, sample=128)   # every token


def test_config2_block_shape_sweep():
    _check_workload(synth.config(2), sample=24)


def test_config3_bert_base_projection_set():
    # all 48 weights built and run; the oracle samples 4 tokens of each
    _check_workload(synth.config(3), sample=4)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shape", [(32, 1), (16, 16)])
def test_config4_bert_large(dtype, shape):
    # first and last layer's Q/K/V/O (8 of 96 weights) at the full 16384 tokens
    wl = synth.config(4, dtype=dtype, shape=shape, only=[0, 1, 2, 3, 92, 93, 94, 95])
    _check_workload(wl, sample=4)


@pytest.mark.parametrize("shape", [(32, 1), (16, 16)])
def test_config5_zipf_rows(shape):
    _check_workload(synth.config(5, shape=shape), sample=6)
