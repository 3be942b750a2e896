"""Entry-range sharding of the lookup: the merge of per-shard results (test infrastructure only).

A store cut into row ranges, shard g holding global entries [base_g, base_g + n_g), can be searched one shard at
a time. The pieces of Algorithm 1's lookup then combine as follows:

* The key check is per entry, so A_q is the disjoint union of the shards' A_q^g (global ids = base_g + local id).
* C_q is the first top_c entries of A_q in (score descending, global id ascending) order. Every member of C_q that
  lives on shard g is among shard g's own first top_c, so C_q is the first top_c of the union of the shards'
  candidate lists under the same order. The bases increase with g, so the tie rule is the same globally.
* A candidate's lookahead scores, token matches and pass bit depend only on its own row and the query.
* The served entry is the first passing member of C_q. The status is HIT, or REJECT when C_q is not empty, or
  MISS_KEY.
* max_j s_qj over all entries is the maximum of the shards' maxima. A shard with candidates has its maximum in
  its first candidate; a shard without reports it as its key score.

merge() applies these rules to the shards' Results. What it returns matches lookup() over the whole store in every
decision and candidate field. It carries no margins, which only the whole-store lookup can compute.
"""
from __future__ import annotations

import numpy as np

from .lookup import HIT, MISS_KEY, REJECT, Params, Result


def merge(results: list, bases: list, params: Params) -> Result:
    """The whole-store Result of a batch from the Results of its shards; bases[g] is shard g's first global id."""
    if len(results) != len(bases) or not results:
        raise ValueError("one base per shard result, at least one shard")
    c = params.top_c
    B = results[0].status.shape[0]
    n_models = results[0].prefix_scores.shape[1]
    out = Result(
        entry_id=np.full(B, -1, np.int32), status=np.full(B, MISS_KEY, np.uint8),
        key_score=np.full(B, -np.inf), prefix_score=np.full(B, np.nan), token_matches=np.full(B, -1, np.int32),
        n_cand=np.zeros(B, np.int32), n_above=np.zeros(B, np.int64),
        cand_id=np.full((B, c), -1, np.int32), cand_score=np.full((B, c), np.nan),
        cand_prefix_score=np.full((B, c), np.nan), cand_matches=np.full((B, c), -1, np.int32),
        prefix_scores=np.full((B, n_models), np.nan),
        cand_pass=np.zeros((B, c), bool), cand_prefix_scores=np.full((B, c, n_models), np.nan),
        margin=np.full(B, np.nan), list_margin=np.full(B, np.nan), literal_margin=np.full(B, np.nan),
        next_id=np.full(B, -1, np.int32), next_score=np.full(B, np.nan))
    for b in range(B):
        pool = []   # (score, global id, shard, slot)
        best = -np.inf
        for g, (res, base) in enumerate(zip(results, bases)):
            nc = int(res.n_cand[b])
            best = max(best, res.cand_score[b, 0] if nc else res.key_score[b])
            out.n_above[b] += res.n_above[b]
            pool += [(res.cand_score[b, i], base + int(res.cand_id[b, i]), g, i) for i in range(nc)]
        pool.sort(key=lambda e: (-e[0], e[1]))
        chosen = pool[:c]
        nc = len(chosen)
        out.n_cand[b] = nc
        out.key_score[b] = best
        for i, (score, gid, g, slot) in enumerate(chosen):
            res = results[g]
            out.cand_id[b, i] = gid
            out.cand_score[b, i] = score
            out.cand_prefix_score[b, i] = res.cand_prefix_score[b, slot]
            out.cand_matches[b, i] = res.cand_matches[b, slot]
            out.cand_pass[b, i] = res.cand_pass[b, slot]
            out.cand_prefix_scores[b, i] = res.cand_prefix_scores[b, slot]
        if not nc:
            continue
        passing = np.nonzero(out.cand_pass[b, :nc])[0]
        shown = int(passing[0]) if passing.size else 0
        if passing.size:
            out.status[b] = HIT
            out.entry_id[b] = out.cand_id[b, shown]
            out.key_score[b] = out.cand_score[b, shown]
        else:
            out.status[b] = REJECT
        out.prefix_score[b] = out.cand_prefix_score[b, shown]
        out.token_matches[b] = out.cand_matches[b, shown]
        out.prefix_scores[b] = out.cand_prefix_scores[b, shown]
    return out
