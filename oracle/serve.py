"""The serve loop around the lookup (test infrastructure only).

Algorithm 1, applied batch by batch. Each query of a batch is checked against the cache as it stood when the
batch began. Then, for every query that was not served (a key miss, or a rejection by the lookahead check),
the query is "decoded from scratch" and its entry ⟨h(x), [h(f_k(x)), f(x)]⟩ is added to the cache. The entries
are appended in query order, and a new entry's id is the next free row.
"""
from __future__ import annotations

import numpy as np

from .lookup import HIT, Params, Result, Store, lookup


class ServeLoop:
    def __init__(self, capacity: int, d: int, k: int, params: Params):
        self.store = Store(np.zeros((capacity, d), np.uint16), np.zeros((capacity, d), np.uint16),
                           np.zeros((capacity, k), np.int32), 0)
        self.params = params

    @property
    def n(self) -> int:
        return self.store.n

    def insert(self, key_bits, prefix_bits, ids) -> int:
        """Append rows; returns the id of the first one."""
        m = len(key_bits)
        first = self.store.n
        if first + m > self.store.key.shape[0]:
            raise OverflowError("cache capacity exceeded")
        self.store.key[first:first + m] = key_bits
        self.store.prefix[first:first + m] = prefix_bits
        self.store.ids[first:first + m] = ids
        self.store.n = first + m
        return first

    def step(self, queries: dict) -> tuple[Result, int, int]:
        """One batch: lookup, then append every query that was not a HIT, in query order."""
        res = lookup(self.store, queries, self.params)
        miss = np.nonzero(res.status != HIT)[0]
        first = self.insert(np.asarray(queries["emb"])[miss], np.asarray(queries["prefix"])[miss],
                            np.asarray(queries["ids"])[miss])
        return res, first, len(miss)
