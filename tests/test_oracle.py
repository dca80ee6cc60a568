"""Pins for the CPU oracle: checks against things other than the oracle itself.

* SciPy's BSR conversion and product (Section 2.2 says the format and the
  sparse multiply follow SciPy), and SciPy's CSR product for 1x1 blocks;
* numpy's float64 matmul of the densified weight, on non-square shapes so a
  transposed operand cannot pass;
* a worked example derived by hand from the definitions;
* invariants: round trips, 0% / 100% sparsity, token permutation, scaling by
  powers of two, block-shape independence, bf16 widening;
* the keep rule's special values (NaN, -0.0, subnormals, ties with thr);
* bfloat16 rounding against torch's conversion and a brute-force table.
"""
import numpy as np
import pytest
import scipy.sparse as sp
import torch

import oracle
import synth

SHAPES = [(1, 1), (4, 4), (8, 1), (16, 1), (32, 1), (1, 32), (16, 16), (32, 32), (2, 3), (3, 2)]


def _block_weight(M, K, R, C, density, seed, dtype="f32"):
    MB, KB = M // R, K // C
    nnzb = int(round(MB * KB * density))
    mask = synth.uniform_block_mask(seed, MB, KB, nnzb)
    W = synth.weight_values(seed, mask, R, C)
    if dtype == "bf16":
        W = synth.to_bf16_bits(W)
    return W, mask


def _f64(a):
    return oracle.widen(a)


# ---------------------------------------------------------------- builder

@pytest.mark.parametrize("R,C", SHAPES)
def test_builder_matches_scipy(R, C):
    M, K = 96, 192
    W, mask = _block_weight(M, K, R, C, 0.3, 11 + R * 7 + C)
    indptr, indices, data = oracle.bsr_from_dense(W, R, C, 0.0)
    ref = sp.bsr_matrix(W, blocksize=(R, C))
    ref.sort_indices()
    assert np.array_equal(indptr, ref.indptr)
    assert np.array_equal(indices, ref.indices)
    assert np.array_equal(data.view(np.uint32), ref.data.astype(np.float32).view(np.uint32))
    assert indptr[-1] == mask.sum()


def test_builder_worked_example():
    # 4x6 weight in 2x3 blocks; blocks (0,1) and (1,0) are all zero.
    W = np.array([[1, 2, 0, 0, 0, 0],
                  [0, 3, 0, 0, 0, 0],
                  [0, 0, 0, 4, 0, 5],
                  [0, 0, 0, 0, 6, 0]], dtype=np.float32)
    indptr, indices, data = oracle.bsr_from_dense(W, 2, 3)
    assert indptr.tolist() == [0, 1, 2]
    assert indices.tolist() == [0, 1]
    assert data.tolist() == [[[1, 2, 0], [0, 3, 0]], [[4, 0, 5], [0, 6, 0]]]
    X = np.array([[1, 1, 1, 1, 1, 1], [1, 2, 3, 4, 5, 6]], dtype=np.float32)
    b = np.array([0.5, -1, 2, 0], dtype=np.float32)
    Y = oracle.bsr_spmm(indptr, indices, data, X, b, 4)
    # row 0: 1+2+0.5, 3-1, 4+5+2, 6 ; row 1: 1+4+0.5, 6-1, 16+30+2, 30
    assert Y.tolist() == [[3.5, 2.0, 11.0, 6.0], [5.5, 5.0, 48.0, 30.0]]


def test_keep_rule_special_values():
    R, C = 2, 2
    nan, tiny = np.float32(np.nan), np.float32(1e-45)   # 1e-45 rounds to the smallest subnormal
    blocks = [
        [[0, 0], [0, 0]],            # all zero: dropped
        [[-0.0, 0], [0, -0.0]],      # negative zeros: dropped
        [[0, nan], [0, 0]],          # NaN: kept
        [[0, 0], [tiny, 0]],         # subnormal: kept at thr = 0
        [[0.25, 0], [0, -0.25]],     # |w| == thr: dropped at thr = 0.25
        [[0, 0], [0, -0.2500001]],   # just above thr: kept at thr = 0.25
    ]
    W = np.zeros((2, 6 * 2), dtype=np.float32)
    for j, blk in enumerate(blocks):
        W[:, 2 * j:2 * j + 2] = np.array(blk, dtype=np.float32)
    _, idx0, _ = oracle.bsr_from_dense(W, R, C, 0.0)
    assert idx0.tolist() == [2, 3, 4, 5]
    _, idx1, data1 = oracle.bsr_from_dense(W, R, C, 0.25)
    assert idx1.tolist() == [2, 5]
    # values inside a kept block are copied bit for bit, sub-threshold ones included
    assert np.array_equal(data1[1].view(np.uint32), W[:, 10:12].view(np.uint32))
    assert np.isnan(data1[0][0, 1])


def test_keep_rule_bf16_widening():
    # bf16 0x0001 is the smallest subnormal: kept at thr=0, dropped at thr=1e-38.
    W = np.zeros((1, 4), dtype=np.uint16)
    W[0, 1] = 0x0001
    W[0, 2] = 0x8000          # -0.0
    W[0, 3] = 0x3F80          # 1.0
    _, idx, data = oracle.bsr_from_dense(W, 1, 1, 0.0)
    assert idx.tolist() == [1, 3] and data.ravel().tolist() == [1, 0x3F80]
    _, idx, _ = oracle.bsr_from_dense(W, 1, 1, 1e-38)
    assert idx.tolist() == [3]
    _, idx, _ = oracle.bsr_from_dense(W, 1, 1, 1.0)
    assert idx.tolist() == []


@pytest.mark.parametrize("R,C", SHAPES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_round_trips(R, C, dtype):
    M, K = 96, 192
    W, _ = _block_weight(M, K, R, C, 0.25, 5 + R + 3 * C, dtype)
    indptr, indices, data = oracle.bsr_from_dense(W, R, C)
    W2 = oracle.bsr_to_dense(indptr, indices, data, M, K)
    assert np.array_equal(W2, W)
    i2, j2, d2 = oracle.bsr_from_dense(W2, R, C)
    assert np.array_equal(i2, indptr) and np.array_equal(j2, indices)
    assert data.tobytes() == d2.tobytes()


def test_builder_threshold_against_brute_force():
    rng = np.random.default_rng(3)
    M, K, R, C = 12, 20, 3, 4
    W = (rng.standard_normal((M, K)) * rng.choice([1e-3, 1.0], size=(M, K))).astype(np.float32)
    thr = 0.5
    indptr, indices, _ = oracle.bsr_from_dense(W, R, C, thr)
    kept = []
    for i in range(M // R):
        for j in range(K // C):
            if any(abs(float(W[i * R + r, j * C + c])) > thr for r in range(R) for c in range(C)):
                kept.append((i, j))
    got = [(i, int(indices[p])) for i in range(M // R) for p in range(indptr[i], indptr[i + 1])]
    assert got == kept


# ---------------------------------------------------------------- product

@pytest.mark.parametrize("R,C", SHAPES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_product_matches_numpy_dense(R, C, dtype):
    M, K, N = 96, 192, 7        # M != K: a transposed operand cannot pass
    W, _ = _block_weight(M, K, R, C, 0.3, 101 + R + C, dtype)
    X = synth.activations(202, N, K, dtype)
    b = synth.normal(303, synth.STREAM_BIAS, M, 0.02)
    bsr = oracle.bsr_from_dense(W, R, C)
    Y = oracle.bsr_spmm(*bsr, X, b, M)
    ref = _f64(X) @ _f64(W).T + b.astype(np.float64)
    E = np.abs(_f64(X)) @ np.abs(_f64(W)).T + np.abs(b.astype(np.float64))
    assert np.all(np.abs(Y - ref) <= 1e-13 * E)
    Eo = oracle.err_bound(*bsr, X, b, M)
    assert np.allclose(Eo, E, rtol=1e-13, atol=0)


@pytest.mark.parametrize("R,C", SHAPES)
def test_product_matches_scipy_bsr(R, C):
    M, K, N = 96, 192, 5
    W, _ = _block_weight(M, K, R, C, 0.2, 77 + R + C)
    X = synth.activations(78, N, K, "f32")
    indptr, indices, data = oracle.bsr_from_dense(W, R, C)
    Y = oracle.bsr_spmm(indptr, indices, data, X, None, M)
    A = sp.bsr_matrix((data.astype(np.float64), indices, indptr), shape=(M, K))
    ref = (A @ X.astype(np.float64).T).T
    E = np.abs(X.astype(np.float64)) @ np.abs(W.astype(np.float64)).T
    assert np.all(np.abs(Y - ref) <= 1e-13 * E)


def test_unit_blocks_match_scipy_csr():
    M, K, N = 64, 80, 6
    W, _ = _block_weight(M, K, 1, 1, 0.2, 9)
    X = synth.activations(10, N, K, "f32")
    bsr = oracle.bsr_from_dense(W, 1, 1)
    Y = oracle.bsr_spmm(*bsr, X, None, M)
    ref = (sp.csr_matrix(W.astype(np.float64)) @ X.astype(np.float64).T).T
    assert np.allclose(Y, ref, rtol=1e-13, atol=1e-15)


def test_block_shape_independence_bitwise():
    # One dense W whose zeros form 32x32 blocks is a valid BSR matrix for every
    # shape dividing 32; the double sum in ascending k is the same number.
    M, K, N = 64, 128, 4
    W, _ = _block_weight(M, K, 32, 32, 0.5, 21)
    X = synth.activations(22, N, K, "f32")
    b = synth.normal(23, synth.STREAM_BIAS, M, 0.02)
    ref = oracle.dense_linear(W, X, b)
    for R, C in [(1, 1), (4, 4), (8, 1), (16, 1), (32, 1), (1, 32), (16, 16), (32, 32), (2, 8)]:
        Y = oracle.bsr_spmm(*oracle.bsr_from_dense(W, R, C), X, b, M)
        assert np.array_equal(Y, ref), (R, C)


def test_zero_sparsity_equals_dense():
    M, K, N = 48, 64, 5
    rng = np.random.default_rng(1)
    W = (rng.standard_normal((M, K)) * 0.02).astype(np.float32)
    W[W == 0] = 1e-3
    X = synth.activations(2, N, K, "f32")
    b = synth.normal(3, synth.STREAM_BIAS, M, 0.02)
    for R, C in [(16, 16), (8, 1), (1, 32)]:
        bsr = oracle.bsr_from_dense(W, R, C)
        assert bsr[0][-1] == (M // R) * (K // C)
        assert np.array_equal(oracle.bsr_spmm(*bsr, X, b, M), oracle.dense_linear(W, X, b))
    ref = X.astype(np.float64) @ W.astype(np.float64).T + b
    assert np.allclose(oracle.dense_linear(W, X, b), ref, rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_full_sparsity_gives_bias(dtype):
    M, K, N = 64, 96, 3
    W = np.zeros((M, K), dtype=np.float32 if dtype == "f32" else np.uint16)
    X = synth.activations(4, N, K, dtype)
    b = synth.normal(5, synth.STREAM_BIAS, M, 0.02)
    indptr, indices, data = oracle.bsr_from_dense(W, 16, 16)
    assert indptr.tolist() == [0] * (M // 16 + 1) and indices.size == 0
    Y = oracle.bsr_spmm(indptr, indices, data, X, b, M)
    assert np.array_equal(Y, np.broadcast_to(b.astype(np.float64), (N, M)))
    assert np.array_equal(oracle.bsr_spmm(indptr, indices, data, X, None, M), np.zeros((N, M)))


def test_token_permutation_and_rows_argument():
    M, K, N = 64, 96, 9
    W, _ = _block_weight(M, K, 8, 1, 0.3, 31)
    X = synth.activations(32, N, K, "f32")
    b = synth.normal(33, synth.STREAM_BIAS, M, 0.02)
    bsr = oracle.bsr_from_dense(W, 8, 1)
    Y = oracle.bsr_spmm(*bsr, X, b, M)
    perm = np.random.default_rng(0).permutation(N)
    assert np.array_equal(oracle.bsr_spmm(*bsr, X[perm], b, M), Y[perm])
    assert np.array_equal(oracle.bsr_spmm(*bsr, X, b, M, rows=perm[:4]), Y[perm[:4]])


def test_power_of_two_scaling():
    M, K, N = 64, 96, 4
    W, _ = _block_weight(M, K, 4, 4, 0.3, 41)
    X = synth.activations(42, N, K, "f32")
    bsr = oracle.bsr_from_dense(W, 4, 4)
    Y = oracle.bsr_spmm(*bsr, X, None, M)
    for k in (-3, 5):
        Xs = (X * np.float32(2.0 ** k)).astype(np.float32)
        assert np.array_equal(oracle.bsr_spmm(*bsr, Xs, None, M), Y * 2.0 ** k)


def test_bf16_inputs_widen_exactly():
    M, K, N = 32, 64, 3
    W, _ = _block_weight(M, K, 16, 16, 0.5, 51, "bf16")
    X = synth.activations(52, N, K, "bf16")
    b = synth.normal(53, synth.STREAM_BIAS, M, 0.02)
    Yb = oracle.bsr_spmm(*oracle.bsr_from_dense(W, 16, 16), X, b, M)
    Wf, Xf = synth.bf16_bits_to_f32(W), synth.bf16_bits_to_f32(X)
    Yf = oracle.bsr_spmm(*oracle.bsr_from_dense(Wf, 16, 16), Xf, b, M)
    assert np.array_equal(Yb, Yf)


# ---------------------------------------------------------------- rounding

def test_round_f32_matches_numpy():
    rng = np.random.default_rng(8)
    x = rng.standard_normal(10000) * 10.0 ** rng.integers(-40, 40, 10000)
    with np.errstate(over="ignore"):   # magnitudes past fp32's range round to inf on purpose
        ref = x.astype(np.float32)
    assert np.array_equal(oracle.round_f32(x).view(np.uint32), ref.view(np.uint32))


def test_round_bf16_matches_torch_on_floats():
    rng = np.random.default_rng(9)
    f = np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * np.float32(2.0) ** rng.integers(-140, 127, 20000),
        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.3895e38, -3.4e38, 1e-45, 9.2e-41],
                 dtype=np.float32),
    ]).astype(np.float32)
    f = f[np.isfinite(f)]
    got = oracle.round_bf16(f.astype(np.float64))
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, ref)


def test_round_bf16_brute_force_on_doubles():
    table = np.arange(0, 0x7F80, dtype=np.uint32)          # every finite non-negative bf16
    vals = (table << 16).view(np.float32).astype(np.float64)
    rng = np.random.default_rng(10)
    x = np.abs(rng.standard_normal(3000)) * 2.0 ** rng.integers(-130, 120, 3000)
    got = oracle.round_bf16(x)
    for xi, gi in zip(x, got):
        k = np.searchsorted(vals, xi)
        lo, hi = max(k - 1, 0), min(k, vals.size - 1)
        dlo, dhi = xi - vals[lo], vals[hi] - xi
        want = lo if dlo < dhi else hi if dhi < dlo else (lo if lo % 2 == 0 else hi)
        assert gi == want, (xi, gi, want)


# ---------------------------------------------------------------- float-accumulate variant (timed baseline)

@pytest.mark.parametrize("R,C", [(32, 1), (16, 16), (1, 1), (1, 32), (3, 2)])
def test_f32acc_exact_on_dyadic_inputs(R, C):
    # small integers scaled by powers of two: every product and partial sum
    # is exact in float, so the float-accumulated product must equal numpy's
    # float64 matmul of the densified weight exactly (non-square: a
    # transposed operand fails)
    M, K, N = 96, 160, 7
    rng = np.random.default_rng(R * 31 + C)
    MB, KB = M // R, K // C
    mask = rng.random((MB, KB)) < 0.35
    W = (rng.integers(-8, 9, size=(M, K)) / 8.0).astype(np.float32)
    W *= np.kron(mask, np.ones((R, C))).astype(np.float32)
    W[W == 0] = 0.0
    X = rng.integers(-16, 17, size=(N, K)).astype(np.float32)
    b = (rng.integers(-4, 5, size=M) / 4.0).astype(np.float32)
    ref = sp.bsr_matrix(W, blocksize=(R, C))
    ref.sort_indices()
    bsr = oracle.bsr_from_dense(W, R, C)
    Y = oracle.bsr_spmm_f32acc(*bsr, X, b, M)
    want = X.astype(np.float64) @ W.astype(np.float64).T + b
    assert Y.dtype == np.float32
    assert np.array_equal(Y.astype(np.float64), want)


def test_f32acc_within_rounding_bound():
    # n float additions of rounded products: |error| <= gamma_(n+1) * sum |x||w|
    # (Higham, Accuracy and Stability of Numerical Algorithms, Sec. 3.1),
    # u = 2^-24, n = terms per output (+1 for the bias)
    R, C, M, K, N = 8, 4, 64, 256, 19
    W, _ = _block_weight(M, K, R, C, 0.4, 901)
    X = synth.activations(902, N, K, "f32")
    b = synth.normal(903, synth.STREAM_BIAS, M, 0.02)
    bsr = oracle.bsr_from_dense(W, R, C)
    Y = oracle.bsr_spmm_f32acc(*bsr, X, b, M).astype(np.float64)
    exact = X.astype(np.float64) @ W.astype(np.float64).T + b
    E = np.abs(X.astype(np.float64)) @ np.abs(W.astype(np.float64)).T + np.abs(b)
    terms = np.diff(bsr[0]).max() * C + 1
    u = 2.0 ** -24
    gamma = (terms + 1) * u / (1 - (terms + 1) * u)
    assert np.all(np.abs(Y - exact) <= gamma * E)
    # and it is not the float64 result rounded once: float accumulation differs somewhere
    assert not np.array_equal(Y, exact.astype(np.float32).astype(np.float64))


def test_f32acc_independent_of_threads_and_tokens():
    R, C, M, K, N = 16, 1, 128, 96, 33
    W, _ = _block_weight(M, K, R, C, 0.5, 911)
    X = synth.activations(912, N, K, "f32")
    b = np.linspace(-0.1, 0.1, M).astype(np.float32)
    bsr = oracle.bsr_from_dense(W, R, C)
    Y1 = oracle.bsr_spmm_f32acc(*bsr, X, b, M, threads=1)
    for t in (2, 3, 8):
        assert np.array_equal(Y1, oracle.bsr_spmm_f32acc(*bsr, X, b, M, threads=t))
    rows = [32, 0, 17]
    assert np.array_equal(Y1[rows], oracle.bsr_spmm_f32acc(*bsr, X, b, M, rows=rows, threads=4))


def test_f32acc_full_sparsity_gives_bias_bf16():
    M, K, R, C = 32, 64, 16, 16
    W = np.zeros((M, K), dtype=np.uint16)
    X = synth.to_bf16_bits(synth.activations(921, 5, K, "f32"))
    b = np.linspace(-1, 1, M).astype(np.float32)
    bsr = oracle.bsr_from_dense(W, R, C)
    assert bsr[0][-1] == 0
    Y = oracle.bsr_spmm_f32acc(*bsr, X, b, M, threads=2)
    assert np.array_equal(Y, np.broadcast_to(b, (5, M)))


# ---------------------------------------------------------------- property

def _divisors(n):
    return [d for d in range(1, n + 1) if n % d == 0]


def _brute_bsr(W, R, C):
    """The three arrays written out from Section 2.2's definition, block by
    block: keep a block iff some element has !(|w| <= 0)."""
    M, K = W.shape
    Wf = W.astype(np.float64)
    indptr, indices, data = [0], [], []
    for i in range(M // R):
        for j in range(K // C):
            blk = Wf[i * R:(i + 1) * R, j * C:(j + 1) * C]
            if np.any(~(np.abs(blk) <= 0.0)):
                indices.append(j)
                data.append(W[i * R:(i + 1) * R, j * C:(j + 1) * C])
        indptr.append(len(indices))
    return indptr, indices, data


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_property_random_tiny_shapes_against_brute_force(dtype):
    """Seeded random cases: M, K <= 64, a block shape (R, C) dividing them,
    block sparsity from 0% to 100% and 1 to 9 tokens. The builder against the
    definition written out block by block (indptr, indices, values bit for
    bit), and the product against explicit sums over the dense weight in
    float64 -- zeros outside the kept blocks add nothing, and the terms come
    in the same ascending column order, so the results agree bit for bit."""
    rng = np.random.default_rng(2106 + (dtype == "bf16"))
    for case in range(60):
        M, K = int(rng.integers(1, 65)), int(rng.integers(1, 65))
        R, C = int(rng.choice(_divisors(M))), int(rng.choice(_divisors(K)))
        density = float(rng.choice([0.0, 0.15, 0.4, 0.8, 1.0]))
        W, _ = _block_weight(M, K, R, C, density, 4000 + case, dtype)
        N = int(rng.integers(1, 10))
        X = synth.activations(5000 + case, N, K, dtype)
        b = synth.normal(6000 + case, 0, M, 0.02).astype(np.float32)
        indptr, indices, data = oracle.bsr_from_dense(W, R, C)
        e_ptr, e_ind, e_data = _brute_bsr(W, R, C)
        assert indptr.tolist() == e_ptr and indices.tolist() == e_ind, (case, M, K, R, C)
        assert data.shape == (len(e_ind), R, C)
        assert all(np.array_equal(data[p].view(np.uint8), np.ascontiguousarray(e_data[p]).view(np.uint8))
                   for p in range(len(e_ind)))
        Y = oracle.bsr_spmm(indptr, indices, data, X, b, M)
        Wd, Xd = _f64(W), _f64(X)
        Yb = np.empty((N, M))
        for n in range(N):
            for m in range(M):
                acc = 0.0
                for k in range(K):
                    acc += Xd[n, k] * Wd[m, k]
                Yb[n, m] = acc + float(b[m])
        assert np.array_equal(Y, Yb), (case, M, K, R, C)
