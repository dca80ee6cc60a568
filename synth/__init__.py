"""Seeded synthetic workloads shaped like the pruned BERT attention projections.

This module only draws inputs: dense weights whose zero pattern is block
structured, activations and biases. It holds none of the arithmetic of the BSR
product or of the BSR conversion; both the CPU oracle tests and the GPU tests
take their inputs from here so that they see identical bytes.

The paper prunes the Q/K/V/O projections of BERT-base (L=12, H=768, A=12,
Section 2.3) into R x C blocks (Eq. 3) and measures block shapes from 1x1 to
64x64 at 80% sparsity (Table 1). Trained weights and the SQuAD/GLUE data are
not available, so every value here is drawn from a seeded generator:

* random bits: splitmix64 (Steele, Lea and Flood, "Fast splittable
  pseudorandom number generators", OOPSLA 2014) evaluated at counter
  positions, so every element is a pure function of (seed, stream, index);
* normals: the Box-Muller transform of two uniforms;
* Zipf(s) variates for uneven rows: Devroye's rejection method
  (Non-Uniform Random Variate Generation, 1986, Ch. X.6).

Sparsity is the fraction of R x C blocks removed. A weight at s% keeps
``(MB*KB*(100-s)+50)//100`` blocks. Weight values are N(0, 0.02) (std), never
exactly zero, so converting the dense weight back to BSR at threshold 0 gives
exactly the drawn block pattern.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional

import numpy as np

_U64 = np.uint64
_GAMMA = _U64(0x9E3779B97F4A7C15)
_M1 = _U64(0xBF58476D1CE4E5B9)
_M2 = _U64(0x94D049BB133111EB)

# Stream identifiers: independent generator streams for each kind of draw.
STREAM_PLACEMENT = 1
STREAM_W = 2
STREAM_X = 3
STREAM_BIAS = 4
STREAM_SPARSITY = 5
STREAM_ZIPF = 6

BASE_SEED = 2106088460

DTYPES = ("f32", "bf16")


def _mix(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> _U64(30))) * _M1
    z = (z ^ (z >> _U64(27))) * _M2
    return z ^ (z >> _U64(31))


def _key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        k = _mix(np.array([(seed * 0x100000001B3 + stream * 0x9E3779B1) & 0xFFFFFFFFFFFFFFFF], dtype=_U64))
    return k[0]


def bits(seed: int, stream: int, start: int, n: int) -> np.ndarray:
    """n uint64 words at counter positions start..start+n-1 of (seed, stream)."""
    return bits_at(seed, stream, np.arange(start, start + n, dtype=_U64))


def bits_at(seed: int, stream: int, positions: np.ndarray) -> np.ndarray:
    """uint64 words at the given counter positions of (seed, stream)."""
    idx = np.asarray(positions).astype(_U64)
    with np.errstate(over="ignore"):
        z = _key(seed, stream) + (idx + _U64(1)) * _GAMMA
        return _mix(z)


def _unit(b: np.ndarray) -> np.ndarray:
    return ((b >> _U64(11)).astype(np.float64) + 1.0) * (1.0 / 9007199254740992.0)


def uniform(seed: int, stream: int, start: int, n: int) -> np.ndarray:
    """Doubles in (0, 1]: the top 53 bits of each word, plus one ulp."""
    return _unit(bits(seed, stream, start, n))


def normal(seed: int, stream: int, n: int, std: float = 1.0, start: int = 0) -> np.ndarray:
    """n draws of N(0, std^2) as float32, none exactly zero (zeros are redrawn)."""
    m = (n + 1) // 2
    u = uniform(seed, stream, 2 * start, 2 * m)
    u1, u2 = u[0::2], u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    th = 2.0 * np.pi * u2
    z = np.empty(2 * m, dtype=np.float64)
    z[0::2] = r * np.cos(th)
    z[1::2] = r * np.sin(th)
    out = (z[:n] * std).astype(np.float32)
    zero = np.flatnonzero(out == 0)
    redraw = 0
    while zero.size:
        redraw += 1
        alt = normal(seed, stream + 1000 * redraw, zero.size, std, start=start + n)
        out[zero] = alt
        zero = np.flatnonzero(out == 0)
    return out


def kept_blocks(MB: int, KB: int, sparsity_pct: float) -> int:
    """Blocks kept at ``sparsity_pct`` percent block sparsity (round half up)."""
    if float(sparsity_pct).is_integer():
        return (MB * KB * (100 - int(sparsity_pct)) + 50) // 100
    return int(np.floor(MB * KB * (100.0 - sparsity_pct) / 100.0 + 0.5))


def uniform_block_mask(seed: int, MB: int, KB: int, nnzb: int) -> np.ndarray:
    """A [MB, KB] bool mask with exactly nnzb True entries, placed uniformly at random."""
    total = MB * KB
    if not 0 <= nnzb <= total:
        raise ValueError("nnzb out of range")
    keys = bits(seed, STREAM_PLACEMENT, 0, total)
    order = np.argsort(keys, kind="stable")
    mask = np.zeros(total, dtype=bool)
    mask[order[:nnzb]] = True
    return mask.reshape(MB, KB)


def zipf_variates(seed: int, n: int, s: float = 1.2) -> np.ndarray:
    """n i.i.d. Zipf(s) integers (s > 1), Devroye's rejection method.

    Variate i uses counter positions of its own, so it does not depend on n.
    Draws above 2**62 are clamped there (they only ever saturate a row).
    """
    if s <= 1.0:
        raise ValueError("Zipf parameter must exceed 1")
    b = 2.0 ** (s - 1.0)
    out = np.zeros(n, dtype=np.float64)
    todo = np.arange(n)
    attempt = 0
    while todo.size:
        base = todo.astype(np.int64) * (1 << 20) + 2 * attempt
        U = _unit(bits_at(seed, STREAM_ZIPF, base))
        V = _unit(bits_at(seed, STREAM_ZIPF, base + 1))
        X = np.floor(U ** (-1.0 / (s - 1.0)))
        X = np.minimum(X, 2.0 ** 62)
        T = (1.0 + 1.0 / X) ** (s - 1.0)
        ok = V * X * (T - 1.0) / (b - 1.0) <= T / b
        out[todo[ok]] = X[ok]
        todo = todo[~ok]
        attempt += 1
        if attempt > 10000:
            raise RuntimeError("Zipf rejection did not terminate")
    return out


def zipf_row_counts(seed: int, MB: int, KB: int, total: int, s: float = 1.2) -> np.ndarray:
    """Per-block-row kept counts with Zipf(s) shape and exact sum ``total``.

    counts_i = min(KB, floor(c * Z_i)) with c the smallest scale (found by
    bisection) whose sum reaches ``total``; any excess is removed one block at
    a time from the largest row that is not full (lowest index on ties), so
    rows that saturate stay fully dense.
    """
    if not 0 <= total <= MB * KB:
        raise ValueError("total out of range")
    Z = zipf_variates(seed, MB, s)

    def counts(c: float) -> np.ndarray:
        return np.minimum(float(KB), np.floor(c * Z)).astype(np.int64)

    lo, hi = 0.0, float(KB) + 1.0
    while counts(hi).sum() < total:
        hi *= 2.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if counts(mid).sum() >= total:
            hi = mid
        else:
            lo = mid
    cnt = counts(hi)
    excess = int(cnt.sum()) - total
    while excess > 0:
        cand = np.where(cnt < KB, cnt, -1)
        if cand.max() <= 0:
            cand = cnt.copy()
        i = int(np.argmax(cand))
        cnt[i] -= 1
        excess -= 1
    return cnt


def mask_from_row_counts(seed: int, counts: np.ndarray, KB: int) -> np.ndarray:
    """Per row i, counts[i] block columns drawn uniformly without replacement."""
    MB = counts.size
    mask = np.zeros((MB, KB), dtype=bool)
    for i in range(MB):
        c = int(counts[i])
        if c == 0:
            continue
        keys = bits(seed, STREAM_PLACEMENT, i * KB, KB)
        mask[i, np.argsort(keys, kind="stable")[:c]] = True
    return mask


def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns (uint16), round to nearest even, via torch."""
    import torch

    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns -> float32 (exact widening)."""
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclasses.dataclass
class Weight:
    """One dense weight W[M, K] whose zeros form an R x C block pattern."""

    name: str
    M: int
    K: int
    R: int
    C: int
    dtype: str
    sparsity: float
    mask: np.ndarray          # [M/R, K/C] bool, the drawn block pattern
    W: np.ndarray             # [M, K] float32, or uint16 bf16 bits
    bias: np.ndarray          # [M] float32

    @property
    def nnzb(self) -> int:
        return int(self.mask.sum())

    @property
    def nnz(self) -> int:
        return self.nnzb * self.R * self.C


def weight_values(seed: int, mask: np.ndarray, R: int, C: int, std: float = 0.02) -> np.ndarray:
    """Dense float32 W: N(0, std) inside kept blocks, exact zeros elsewhere."""
    MB, KB = mask.shape
    W = np.zeros((MB, R, KB, C), dtype=np.float32)
    bi, bj = np.nonzero(mask)
    vals = normal(seed, STREAM_W, bi.size * R * C, std).reshape(bi.size, R, C)
    W[bi, :, bj, :] = vals
    return W.reshape(MB * R, KB * C)


def make_weight(name: str, seed: int, M: int, K: int, R: int, C: int, dtype: str,
                sparsity: float, mask: Optional[np.ndarray] = None, std: float = 0.02) -> Weight:
    if M % R or K % C:
        raise ValueError("M and K must be multiples of R and C")
    MB, KB = M // R, K // C
    if mask is None:
        mask = uniform_block_mask(seed, MB, KB, kept_blocks(MB, KB, sparsity))
    W = weight_values(seed, mask, R, C, std)
    bias = normal(seed, STREAM_BIAS, M, std)
    if dtype == "bf16":
        W = to_bf16_bits(W)
    elif dtype != "f32":
        raise ValueError(dtype)
    return Weight(name, M, K, R, C, dtype, sparsity, mask, W, bias)


def activations(seed: int, N: int, K: int, dtype: str) -> np.ndarray:
    """X[N, K] with N(0, 1) entries, float32 or bf16 bits."""
    x = normal(seed, STREAM_X, N * K, 1.0).reshape(N, K)
    return to_bf16_bits(x) if dtype == "bf16" else x


def config_seed(config: int, weight_index: int = 0, shape_index: int = 0) -> int:
    return BASE_SEED + 1000 * config + 10 * weight_index + shape_index


SWEEP_SHAPES = [(1, 1), (4, 4), (8, 1), (16, 1), (32, 1), (1, 32), (16, 16), (32, 32)]
SPARSITY_CHOICES = (50, 70, 80, 90, 95)


@dataclasses.dataclass
class Workload:
    """A set of weights that share one activation matrix X[N, K]."""

    name: str
    N: int
    K: int
    dtype: str
    weights: List[Weight]
    X: Optional[np.ndarray] = None
    seed: int = 0

    def make_X(self, N: Optional[int] = None) -> np.ndarray:
        return activations(self.seed, self.N if N is None else N, self.K, self.dtype)

    @property
    def flops(self) -> int:
        return sum(2 * self.N * w.nnz for w in self.weights)


def sweep_sparsities(n_weights: int, config: int = 3) -> List[int]:
    u = uniform(config_seed(config), STREAM_SPARSITY, 0, n_weights)
    return [SPARSITY_CHOICES[min(4, int(x * 5.0 - 1e-12))] for x in u]


def config(k: int, dtype: Optional[str] = None, shape: Optional[tuple] = None,
           n_weights: Optional[int] = None, N: Optional[int] = None,
           only: Optional[List[int]] = None) -> Workload:
    """The five benchmark workloads (1-based ``k``), optionally cut down.

    1: one 768x768 fp32 weight, 32x1 blocks, 90%; X 128x768.
    2: 768x768 fp32 at 80% for each shape in SWEEP_SHAPES; X 1024x768.
    3: 48 weights (12 layers x Q,K,V,O) 768x768 fp32, 32x1, sparsity drawn
       from {50,70,80,90,95}%; X 1024x768.
    4: 96 weights (24 layers x Q,K,V,O) 1024x1024 at 90%, 32x1 or 16x16;
       X 16384x1024, fp32 or bf16.
    5: one 4096x4096 bf16 weight at 95% with Zipf(1.2) rows, 32x1 or 16x16;
       X 8192x4096 bf16.

    ``only`` keeps just the listed weight indices of workloads 3 and 4.
    """
    if k == 1:
        s = config_seed(1)
        w = make_weight("cfg1_32x1", s, 768, 768, 32, 1, "f32", 90)
        return Workload("cfg1", N or 128, 768, "f32", [w], seed=s)
    if k == 2:
        ws = []
        for si, (R, C) in enumerate(SWEEP_SHAPES):
            if shape is not None and (R, C) != tuple(shape):
                continue
            ws.append(make_weight(f"cfg2_{R}x{C}", config_seed(2, 0, si), 768, 768, R, C, "f32", 80))
        return Workload("cfg2", N or 1024, 768, "f32", ws, seed=config_seed(2))
    if k == 3:
        nw = 48 if n_weights is None else n_weights
        sp = sweep_sparsities(48)
        ids = range(nw) if only is None else only
        ws = [make_weight(f"cfg3_L{i // 4}_{'QKVO'[i % 4]}", config_seed(3, i), 768, 768, 32, 1, "f32", sp[i])
              for i in ids]
        return Workload("cfg3", N or 1024, 768, "f32", ws, seed=config_seed(3))
    if k == 4:
        dt = dtype or "f32"
        R, C = shape or (32, 1)
        si = 0 if (R, C) == (32, 1) else 1
        nw = 96 if n_weights is None else n_weights
        ids = range(nw) if only is None else only
        ws = [make_weight(f"cfg4_L{i // 4}_{'QKVO'[i % 4]}_{R}x{C}", config_seed(4, i, si), 1024, 1024, R, C, dt, 90)
              for i in ids]
        return Workload(f"cfg4_{dt}", N or 16384, 1024, dt, ws, seed=config_seed(4, 0, 9))
    if k == 5:
        R, C = shape or (32, 1)
        si = 0 if (R, C) == (32, 1) else 1
        s = config_seed(5, 0, si)
        MB, KB = 4096 // R, 4096 // C
        cnt = zipf_row_counts(s, MB, KB, kept_blocks(MB, KB, 95))
        mask = mask_from_row_counts(s, cnt, KB)
        w = make_weight(f"cfg5_{R}x{C}", s, 4096, 4096, R, C, "bf16", 95, mask=mask)
        return Workload("cfg5", N or 8192, 4096, "bf16", [w], seed=config_seed(5, 0, 9))
    raise ValueError(f"no workload {k}")
