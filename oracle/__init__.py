"""Oracle for the LaCache two-stage lookahead lookup: plain, slow, fp64, on the CPU.

This package is test infrastructure. Only the tests, the smoke check and the benchmark's CPU-baseline leg may
import it. The CUDA library shares no code with it and never calls it.

Every function here is pinned by tests against values fixed by the paper or by mathematics. The pins are exact
dyadic dot products, hand-built decisions, brute force in exact rational arithmetic, library special cases and
the counts of the paper's Table 3.
"""
from .bf16 import round_to_bf16, widen
from .lookup import (CHECK_BOTH, CHECK_EMB, CHECK_TOKENS, HIT, MISS_KEY, REJECT, KeyCheck, Params, Result,
                     Store, decide, lookahead, lookup, passes)
from .serve import ServeLoop
from .calibrate import calibrate, nearest_rank, pair_similarities
from .lsh import LshKeyCheck, hamming, lookup_lsh, projections, signatures
from .speculative import accepted_prefix
from .shards import merge as merge_shards

__all__ = ["round_to_bf16", "widen", "CHECK_BOTH", "CHECK_EMB", "CHECK_TOKENS", "HIT", "MISS_KEY", "REJECT",
           "KeyCheck", "Params", "Result", "Store", "decide", "lookahead", "lookup", "passes", "ServeLoop",
           "calibrate", "nearest_rank", "pair_similarities", "LshKeyCheck", "hamming", "lookup_lsh", "projections", "signatures",
           "accepted_prefix", "merge_shards"]
