"""The seeded generator: determinism, exact block counts, workload shapes,
and the frozen structures in tests/golden/structures.json."""
import json
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "structures.json")


def test_bits_are_counter_based():
    a = synth.bits(7, 1, 0, 100)
    b = synth.bits(7, 1, 40, 20)
    assert np.array_equal(a[40:60], b)
    assert not np.array_equal(synth.bits(7, 2, 0, 100), a)
    assert len(set(a.tolist())) == 100


def test_normal_moments_and_no_zeros():
    z = synth.normal(1, synth.STREAM_X, 200001, 1.0)
    assert z.dtype == np.float32 and np.all(z != 0)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1.0) < 0.01
    w = synth.normal(2, synth.STREAM_W, 100000, 0.02)
    assert abs(w.std() - 0.02) < 0.0005


@pytest.mark.parametrize("MB,KB,s", [(24, 768, 90), (768, 768, 80), (48, 48, 80), (32, 1024, 90), (4, 4, 50)])
def test_uniform_mask_exact_count(MB, KB, s):
    m = synth.uniform_block_mask(5, MB, KB, synth.kept_blocks(MB, KB, s))
    assert m.shape == (MB, KB)
    assert m.sum() == (MB * KB * (100 - s) + 50) // 100


def test_uniform_mask_is_spread():
    m = synth.uniform_block_mask(9, 24, 768, 3686)
    per_row = m.sum(1)
    assert per_row.min() > 110 and per_row.max() < 200


def test_zipf_rows():
    for (MB, KB, total) in [(128, 4096, 26214), (256, 256, 3277)]:
        cnt = synth.zipf_row_counts(123, MB, KB, total)
        assert cnt.sum() == total and cnt.max() <= KB and cnt.min() >= 0
        assert (cnt == 0).sum() > MB // 2          # many empty rows
        assert (cnt == KB).sum() >= 1               # some dense rows


def test_zipf_variates_distribution():
    z = synth.zipf_variates(77, 20000, 1.2)
    assert z.min() >= 1
    # P(Z = 1) = 1 / zeta(1.2) ~= 0.1815
    assert abs((z == 1).mean() - 0.1815) < 0.012
    assert abs((z == 2).mean() - 0.1815 * 2 ** -1.2) < 0.01


def test_weight_values_respect_mask():
    wl = synth.config(2, shape=(16, 16))
    w = wl.weights[0]
    blocks = (w.W.reshape(w.M // 16, 16, w.K // 16, 16) != 0).any(axis=(1, 3))
    assert np.array_equal(blocks, w.mask)
    assert (w.W.reshape(w.M // 16, 16, w.K // 16, 16) != 0).all(axis=(1, 3))[w.mask].all()


def test_bf16_bits_roundtrip():
    x = synth.normal(3, synth.STREAM_X, 1000)
    b = synth.to_bf16_bits(x)
    assert b.dtype == np.uint16
    assert np.array_equal(synth.to_bf16_bits(synth.bf16_bits_to_f32(b)), b)
    assert np.all(np.abs(synth.bf16_bits_to_f32(b) - x) <= np.abs(x) * 2.0 ** -8)


def test_workload_shapes():
    assert [w.nnzb for w in synth.config(1).weights] == [1843]
    assert [(w.R, w.C) for w in synth.config(2).weights] == synth.SWEEP_SHAPES
    wl4 = synth.config(4, dtype="bf16", shape=(16, 16), n_weights=2, N=16)
    assert wl4.weights[0].nnzb == 410 and wl4.weights[0].W.dtype == np.uint16
    assert synth.config(4, n_weights=1, N=16).weights[0].nnzb == 3277
    assert set(synth.sweep_sparsities(48)) <= set(synth.SPARSITY_CHOICES)


def test_golden_structures():
    import oracle
    from tests.golden.make_golden import build
    with open(GOLDEN) as f:
        want = json.load(f)
    assert build() == want
