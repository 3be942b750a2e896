"""Draft verification for reusing the lookahead prefix on a miss (test infrastructure only).

Section 3.3 ("Speculative Decoding"): when a query is not served from the cache, its k draft tokens f_k(x),
already decoded for the lookahead check, are verified by the target model f in one forward pass. From the
first token on, draft token t is accepted if P_f(t) >= P_g(t), where P_f and P_g are the probabilities the
target and the draft assign to it. The first rejected token ends the reuse, and f decodes from there. The
tokens reused for a query are its accepted prefix: the number of leading positions that pass. A served query
(HIT) decodes nothing, so none of its tokens are verified (-1).
"""
from __future__ import annotations

import numpy as np

from .lookup import HIT


def accepted_prefix(p_target, p_draft, status=None) -> np.ndarray:
    """Per query: the number of leading draft tokens with P_f >= P_g; -1 for a HIT when status is given."""
    pf = np.asarray(p_target, dtype=np.float64)
    pg = np.asarray(p_draft, dtype=np.float64)
    B, k = pf.shape
    out = np.empty(B, dtype=np.int32)
    for b in range(B):
        n = 0
        while n < k and pf[b, n] >= pg[b, n]:
            n += 1
        out[b] = n
    if status is not None:
        out[np.asarray(status) == HIT] = -1
    return out
