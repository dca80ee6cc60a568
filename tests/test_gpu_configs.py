"""The five benchmark workloads at full size, through the C ABI in the launch
configuration the benchmark uses. For every weight the builder is checked bit
for bit against the oracle, and the product on a sample of tokens (first,
last and seeded random ones) plus one whole 128-token tile from the middle of
N (a tile of the full-size launch: its CTA count, task sizes and waves differ
from the small tests'); at least one weight of every kernel configuration the
workloads launch is checked on every token."""
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


def _middle_tile(N, tile=128):
    start = max(0, (N // 2) // tile * tile)
    return np.arange(start, min(N, start + tile))


def _check_workload(wl, sample=12, full=()):
    """`full`: indices of weights checked on every token."""
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
        if i in full:
            rows = None
        else:
            rows = np.union1d(_sample_rows(wl.N, sample, 17 + i), _middle_tile(wl.N))
        check_product(Yh, ref, X, w.bias, w.M, rows=rows)
        h.destroy()


def test_config1_bert_base_single_weight():
    wl = synth.config(1)
    _check_workload(wl, sample=128)   # every token


def test_config2_block_shape_sweep():
    wl = synth.config(2)
    _check_workload(wl, full=range(len(wl.weights)))   # every shape, every token


def test_config3_bert_base_projection_set():
    # all 48 weights built and run; the oracle checks 4 sampled tokens and a
    # middle tile of each, and every token of one weight per sparsity level
    wl = synth.config(3)
    sp = synth.sweep_sparsities(48)
    full = {sp.index(s) for s in set(sp)}
    _check_workload(wl, sample=4, full=full)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shape", [(32, 1), (16, 16)])
def test_config4_bert_large(dtype, shape):
    # first and last layer's Q/K/V/O (8 of 96 weights) at the full 16384
    # tokens; the first on every token
    wl = synth.config(4, dtype=dtype, shape=shape, only=[0, 1, 2, 3, 92, 93, 94, 95])
    _check_workload(wl, sample=4, full={0})


@pytest.mark.parametrize("shape", [(32, 1), (16, 16)])
def test_config5_zipf_rows(shape):
    _check_workload(synth.config(5, shape=shape), full={0})
