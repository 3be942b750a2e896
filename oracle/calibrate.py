"""Threshold calibration (test infrastructure only).

App. A.2 ("Threshold Calibration") sets the two thresholds from benign paraphrase pairs (x, x'):
    tau_c = min(0.80, P5  of sim(emb(x), emb(x')))                 (key check)
    tau_a = min(0.70, P10 of sim(emb(f_k(x)), emb(f_k(x'))))       (lookahead check, per embedding model)
The paper does not state how its percentiles interpolate. The reading here is the nearest-rank percentile: the
P-th percentile of n values is the value of rank ceil(P/100 * n) in ascending order (rank 1 is the smallest,
and P = 0 gives rank 1).
"""
from __future__ import annotations

import math

import numpy as np

from .bf16 import widen


def pair_similarities(x_bits, y_bits) -> np.ndarray:
    """sim of each pair: the dot product of two unit-norm bf16 embeddings, widened exactly to fp64."""
    return np.einsum("ij,ij->i", widen(x_bits), widen(y_bits))


def nearest_rank(values, percentile: float):
    v = np.sort(np.asarray(values, dtype=np.float64))
    if v.size == 0:
        raise ValueError("no values")
    rank = max(1, math.ceil(percentile / 100.0 * v.size))
    return v[min(rank, v.size) - 1]


def calibrate(x_bits, y_bits, percentile: float, cap: float):
    """(threshold, percentile value): min(cap, P-th percentile of the pair similarities)."""
    p = nearest_rank(pair_similarities(x_bits, y_bits), percentile)
    return min(cap, p), p
