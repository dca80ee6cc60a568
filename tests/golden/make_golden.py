"""Writes tests/golden/structures.json from the seeded generator and the CPU oracle.

The paper prints no worked example of a BSR product, so these fixtures freeze
what the generator and the oracle produce for the benchmark workloads: block
structures (indptr/indices hashes, empty and dense block rows) and the
oracle's float64 output for the first tokens of the 768x768 32x1 case. Only
``synth`` and ``oracle`` are called.

    python tests/golden/make_golden.py
"""
import hashlib
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "structures.json")


def sha(a: np.ndarray) -> str:
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).hexdigest()


def describe(w: synth.Weight) -> dict:
    indptr, indices, _ = oracle.bsr_from_dense(w.W, w.R, w.C, 0.0)
    counts = np.diff(indptr)
    return {
        "name": w.name, "M": w.M, "K": w.K, "R": w.R, "C": w.C, "dtype": w.dtype,
        "nnzb": int(indptr[-1]), "empty_rows": int((counts == 0).sum()),
        "dense_rows": int((counts == w.K // w.C).sum()),
        "indptr_sha256": sha(indptr), "indices_sha256": sha(indices),
    }


def build() -> dict:
    out = {"weights": [], "cfg3_sparsities": synth.sweep_sparsities(48)}
    wl1 = synth.config(1)
    out["weights"].append(describe(wl1.weights[0]))
    for w in synth.config(2).weights:
        out["weights"].append(describe(w))
    for w in synth.config(3, n_weights=4).weights:
        out["weights"].append(describe(w))
    for shape in [(32, 1), (16, 16)]:
        out["weights"].append(describe(synth.config(5, shape=shape).weights[0]))
    w = wl1.weights[0]
    X = wl1.make_X()
    Y = oracle.bsr_spmm(*oracle.bsr_from_dense(w.W, w.R, w.C), X, w.bias, w.M, rows=np.arange(8))
    out["cfg1_first8_tokens_Y_float64_sha256"] = sha(Y)
    return out


if __name__ == "__main__":
    with open(OUT, "w") as f:
        json.dump(build(), f, indent=1)
    print("wrote", OUT)
