"""LSH-key variant of the key check (test infrastructure only).

Section 2 assumes an indexing scheme h(.) over the embedding with the gapped-LSH property of Eq. 1: keys of close
embeddings collide with probability above p1, keys of distant ones below p2. Algorithm 1 searches the cache with
that key. The index here is random-hyperplane LSH (SimHash): with b hyperplanes r_1..r_b, the signature of z has
bit i set iff <r_i, z> >= 0. For two embeddings at angle theta each bit agrees with probability 1 - theta/pi, the
published collision probability of this family. Cosine distance is monotone in theta, so it is a gapped LSH for
cosine distance.

The lookup with this index keeps only the entries whose signatures are within Hamming distance `radius` of the
query's (the index's "hit"), then applies the exact key check to them:
    A_q = {j : hamming(sig(q), sig(K_j)) <= radius and sim(q, K_j) >= tau_c}
Stage 2 and the decision are unchanged. With radius >= b nothing is pruned and this is the exact lookup.

A signature bit is a floating-point sign decision. A bit whose projection lies within `amb` of zero is
ambiguous: fp32 and fp64 may disagree on it. The oracle reports those bits so that the comparison can
exclude entries whose inclusion they could flip.
"""
from __future__ import annotations

import numpy as np

from .bf16 import widen
from .lookup import KeyCheck, Params, Store, decide

AMBIGUOUS = 1e-4


def projections(rows_bits, hyperplanes_bits) -> np.ndarray:
    """<r_i, z> for every row z and hyperplane r_i, fp64 from the exact bf16 values: [rows, b]."""
    return widen(rows_bits) @ widen(hyperplanes_bits).T


def signatures(rows_bits, hyperplanes_bits, amb: float = AMBIGUOUS):
    """(bits [rows, b] bool, ambiguous [rows, b] bool): bit i is set iff <r_i, z> >= 0."""
    p = projections(rows_bits, hyperplanes_bits)
    return p >= 0.0, np.abs(p) < amb


def hamming(a_bits, b_bits) -> np.ndarray:
    """Hamming distances between every signature of a [n, b] and every one of b [m, b]: [n, m]."""
    a = np.asarray(a_bits, dtype=np.float64)
    b = np.asarray(b_bits, dtype=np.float64)
    # bits differ where exactly one is set: a + b - 2ab summed over the bits (counts of at most b bits: integers,
    # exact in fp64, which lets the product run as a library matrix product)
    return np.rint(a.sum(axis=1)[:, None] + b.sum(axis=1)[None, :] - 2 * (a @ b.T)).astype(np.int64)


class LshKeyCheck:
    """The key check with the SimHash index as the cache search, fed block by block like KeyCheck: of each block
    of entries, those whose signature is within `radius` of the query's are admitted to the exact check.

    `kc` is the underlying KeyCheck (decide() takes it); ambiguous[q] is True if ambiguous signature bits of the
    query or of an entry could move an entry with sim >= tau_c - 2e-3 across the Hamming radius."""

    def __init__(self, q_bits, tau_c: float, hyperplanes_bits, radius: int):
        self.hyperplanes_bits, self.radius = hyperplanes_bits, radius
        self.q_sig, self.q_amb = signatures(q_bits, hyperplanes_bits)
        self.kc = KeyCheck(q_bits, tau_c)
        self.ambiguous = np.zeros(self.q_sig.shape[0], dtype=bool)

    def add_rows(self, key_bits, j0: int) -> None:
        e_sig, e_amb = signatures(key_bits, self.hyperplanes_bits)
        hd = hamming(self.q_sig, e_sig)
        s = self.kc.q @ widen(key_bits).T
        slack = self.q_amb.sum(axis=1)[:, None] + e_amb.sum(axis=1)[None, :]
        near = s >= self.kc.tau_c - 2e-3
        self.ambiguous |= np.any(near & (slack > 0) & (np.abs(hd - self.radius) <= slack), axis=1)
        self.kc.add_scores(s, j0, admitted=hd <= self.radius)


def lookup_lsh(store: Store, queries: dict, params: Params, hyperplanes_bits, radius: int,
               block_rows: int = 1 << 15):
    """Algorithm 1's two checks with the SimHash index as the cache search.

    Returns (Result, ambiguous): ambiguous[q] is True if ambiguous signature bits of the query or of an entry
    could move an entry with sim >= tau_c - 2e-3 across the Hamming radius."""
    lk = LshKeyCheck(queries["emb"], params.tau_c, hyperplanes_bits, radius)
    for j0 in range(0, store.n, block_rows):
        lk.add_rows(store.key[j0:min(store.n, j0 + block_rows)], j0)
    res = decide(lk.kc, queries["prefix"], queries["ids"], params, lambda j: store.prefix[j],
                 lambda j: store.ids[j])
    return res, lk.ambiguous
