"""Plain fp64 statement of the two-stage lookahead lookup (test infrastructure only).

What is computed, and where the paper states it:

* The cache entry is ⟨h(x), [h(f_k(x)), f(x)]⟩ (§3.2 "Cache Structure"). Here that is a key embedding, the
  embedding of the first k response tokens, and those k token ids. The entry id stands for f(x).
* A query x is served from entry x' only if both checks hold (Algorithm 1; §4.1 "Metrics"):
    stage 1, key check:        sim(x, x')          >= tau_c
    stage 2, lookahead check:  sim(f_k(x), f_k(x')) >= tau_a
  Otherwise x is decoded from scratch and its entry is added to the cache (Algorithm 1, last two steps).
* sim is cosine similarity. The embeddings are unit vectors, so it is their inner product. The oracle takes
  the plain dot product of the stored bf16 values, widened exactly to fp64, with no re-normalisation.

Readings where the paper leaves the batched form open:

* "Search the cache" yields C_q: the top_c entries with s_qj >= tau_c, ordered by score descending, then entry id
  ascending (the older entry first).
* Stage 2 examines C_q in that order. The served entry j* is the first candidate that passes.
* Status per query: HIT (j* exists), REJECT (candidates, none pass), or MISS_KEY (no entry clears tau_c).
* Check modes. EMB: r >= tau_a, the evaluated form (§4.1). TOKENS: at least ``token_match_min`` of the k prefix
  token ids are equal position by position; with token_match_min = k this is Algorithm 1's literal equality
  h(f_k(x')) = h(f_k(x)) under an identity hash on ids. BOTH: both.

Beside the decision the oracle emits two margins per query. The decision margin is the smallest distance by which
some score would have to move to change the status or the served entry: while every key and prefix score moves by
less than half of it, the decision stays as it is. The list margin is the same for the candidate list and its
order. A fp32 implementation may legitimately differ from this fp64 one only where the corresponding margin is
small.
"""
from __future__ import annotations

import dataclasses
from typing import Callable

import numpy as np

from .bf16 import widen

MISS_KEY, HIT, REJECT = 0, 1, 2
CHECK_EMB, CHECK_TOKENS, CHECK_BOTH = 0, 1, 2


@dataclasses.dataclass(frozen=True)
class Params:
    tau_c: float
    tau_a: float
    top_c: int
    check_mode: int = CHECK_EMB
    token_match_min: int | None = None     # None: all k ids must match
    # Ensemble of m lookahead checks (section 3.4, "Analysis"): the prefix row holds one embedding per model,
    # segments of these dimensions, each with its own threshold. None: a single check with tau_a over the row.
    prefix_dims: tuple | None = None
    tau_a_models: tuple | None = None

    def segments(self, row_len: int):
        """(start, end, threshold) of each lookahead check over a prefix row of row_len values."""
        if self.prefix_dims is None:
            return [(0, row_len, self.tau_a)]
        out, start = [], 0
        for dim, tau in zip(self.prefix_dims, self.tau_a_models):
            out.append((start, start + dim, tau))
            start += dim
        if start != row_len:
            raise ValueError(f"prefix dims {self.prefix_dims} do not add up to the row length {row_len}")
        return out


@dataclasses.dataclass
class Store:
    """Entries as three row-aligned arrays; entry id = row index. Rows [0, n) are valid.

    key:    uint16 [cap, d]  bf16 bit patterns of h(x)'s embedding
    prefix: uint16 [cap, d]  bf16 bit patterns of the k-token prefix embedding, h(f_k(x))
    ids:    int32  [cap, k]  the k prefix token ids f_k(x)
    """
    key: np.ndarray
    prefix: np.ndarray
    ids: np.ndarray
    n: int

    @staticmethod
    def of(key, prefix, ids) -> "Store":
        key = np.ascontiguousarray(key, dtype=np.uint16)
        return Store(key, np.ascontiguousarray(prefix, dtype=np.uint16),
                     np.ascontiguousarray(ids, dtype=np.int32), key.shape[0])


@dataclasses.dataclass
class Result:
    entry_id: np.ndarray          # int32 [B]; -1 unless HIT
    status: np.ndarray            # uint8 [B]; MISS_KEY / HIT / REJECT
    key_score: np.ndarray         # f64 [B]; s of j* on HIT, else max_j s_qj (-inf for an empty cache)
    prefix_score: np.ndarray      # f64 [B]; r of j* on HIT, r of the first candidate on REJECT, NaN on MISS_KEY
    token_matches: np.ndarray     # int32 [B]; m of the same candidate as prefix_score, -1 on MISS_KEY
    n_cand: np.ndarray            # int32 [B]; |C_q|
    n_above: np.ndarray           # int64 [B]; |A_q| = #{j : s_qj >= tau_c}
    cand_id: np.ndarray           # int32 [B, c]; C_q in order, -1 padded
    cand_score: np.ndarray        # f64 [B, c]; s, NaN padded
    cand_prefix_score: np.ndarray  # f64 [B, c]; r, NaN padded
    cand_matches: np.ndarray      # int32 [B, c]; m, -1 padded
    prefix_scores: np.ndarray     # f64 [B, models]; every model's r for the candidate of prefix_score
    cand_pass: np.ndarray         # bool [B, c]; each candidate passes the lookahead check (False padded)
    cand_prefix_scores: np.ndarray  # f64 [B, c, models]; every model's r per candidate, NaN padded
    margin: np.ndarray            # f64 [B]; decision margin: smallest score change altering status/entry_id
    list_margin: np.ndarray       # f64 [B]; smallest score change altering C_q or its order
    literal_margin: np.ndarray    # f64 [B]; min(|max_j s - tau_c|, s_(1) - s_(2))
    next_id: np.ndarray           # int32 [B]; the (c+1)-th entry of A_q, -1 if none
    next_score: np.ndarray        # f64 [B]; its score, NaN if none


class KeyCheck:
    """Stage 1 over the store, one block of rows at a time.

    s_qj = <q, K_j> for every valid entry j, in fp64 from the exact bf16 values. A_q = {j : s_qj >= tau_c} is
    the union of the blocks' contributions, so the blocks can come from anywhere: a resident array, or chunks
    regenerated one at a time for a cache larger than host memory. Alongside A_q it keeps max_j s_qj,
    min_j |s_qj - tau_c| and the best score below tau_c, which the margin needs.
    """

    def __init__(self, q_bits, tau_c: float):
        self.q = widen(q_bits)
        self.tau_c = float(tau_c)
        B = self.q.shape[0]
        self._s = [[] for _ in range(B)]
        self._j = [[] for _ in range(B)]
        self.best = np.full(B, -np.inf)
        self.closest = np.full(B, np.inf)
        self.below = np.full(B, -np.inf)
        self.rows = 0

    def add_rows(self, key_bits, j0: int) -> None:
        K = widen(key_bits)
        if K.shape[0] == 0:
            return
        self.add_scores(self.q @ K.T, j0)

    def add_scores(self, s, j0: int, admitted=None) -> None:
        """Fold the scores s [B, rows] of rows j0.. into A_q. With an index, only the rows it admits
        (admitted [B, rows] True) are searched at all; the others count for nothing."""
        if s.shape[1] == 0:
            return
        ok = np.ones(s.shape, dtype=bool) if admitted is None else admitted
        for b in range(s.shape[0]):
            sel = np.nonzero(ok[b] & (s[b] >= self.tau_c))[0]
            if sel.size:
                self._s[b].append(s[b, sel])
                self._j[b].append(sel.astype(np.int64) + j0)
        self.best = np.maximum(self.best, np.where(ok, s, -np.inf).max(axis=1))
        self.closest = np.minimum(self.closest, np.where(ok, np.abs(s - self.tau_c), np.inf).min(axis=1))
        self.below = np.maximum(self.below, np.where(ok & (s < self.tau_c), s, -np.inf).max(axis=1))
        self.rows += s.shape[1]

    def above(self, b: int):
        """A_q for query b, ordered by (score descending, entry id ascending)."""
        if not self._s[b]:
            return np.empty(0), np.empty(0, dtype=np.int64)
        s = np.concatenate(self._s[b])
        j = np.concatenate(self._j[b])
        order = np.lexsort((j, -s))
        return s[order], j[order]


def lookahead(p_bits, t_ids, cand_prefix_bits, cand_ids, segments=None):
    """Stage 2 for one query against the prefix rows of its candidates.

    r_j = <p, P_j>, the cosine similarity sim(f_k(x), f_k(x')) of the two prefix embeddings; with an ensemble,
    one such similarity per model over that model's segment of the row (columns of r).
    m_j = #{i < k : t_i = T_ji}, the positions where the two k-token prefixes carry the same token id.
    """
    P = widen(cand_prefix_bits)
    p = widen(p_bits)
    if segments is None:
        r = P @ p
    else:
        r = np.stack([P[:, a:b] @ p[a:b] for a, b, _ in segments], axis=1)
    m = (np.asarray(cand_ids, dtype=np.int64) == np.asarray(t_ids, dtype=np.int64)[None, :]).sum(axis=1)
    return r, m


def passes(r, m, params: Params, k: int, segments=None):
    """Pass bits of the candidates. With an ensemble, the lookahead check passes only if every model's
    similarity clears that model's threshold (section 3.4: all m checks must hold)."""
    tmin = k if params.token_match_min is None else params.token_match_min
    if segments is None:
        emb_ok = r >= params.tau_a
    else:
        emb_ok = np.all(r >= np.array([t for _, _, t in segments])[None, :], axis=1)
    tok_ok = m >= tmin
    if params.check_mode == CHECK_EMB:
        return emb_ok
    if params.check_mode == CHECK_TOKENS:
        return tok_ok
    if params.check_mode == CHECK_BOTH:
        return emb_ok & tok_ok
    raise ValueError(f"unknown check mode {params.check_mode}")


def decide(kc: KeyCheck, q_prefix_bits, q_ids, params: Params,
           prefix_rows: Callable, id_rows: Callable) -> Result:
    """Candidate selection, stage 2 and the decision for every query of the batch."""
    q_ids = np.asarray(q_ids, dtype=np.int32)
    B = kc.q.shape[0]
    k = q_ids.shape[1]
    segs = params.segments(np.asarray(q_prefix_bits).shape[1]) if params.prefix_dims is not None else None
    n_models = len(segs) if segs else 1
    c = params.top_c
    tau_c, tau_a = params.tau_c, params.tau_a
    uses_r = params.check_mode in (CHECK_EMB, CHECK_BOTH)
    uses_m = params.check_mode in (CHECK_TOKENS, CHECK_BOTH)
    tmin = k if params.token_match_min is None else params.token_match_min

    res = Result(
        entry_id=np.full(B, -1, np.int32), status=np.full(B, MISS_KEY, np.uint8),
        key_score=kc.best.copy(), prefix_score=np.full(B, np.nan), token_matches=np.full(B, -1, np.int32),
        n_cand=np.zeros(B, np.int32), n_above=np.zeros(B, np.int64),
        cand_id=np.full((B, c), -1, np.int32), cand_score=np.full((B, c), np.nan),
        cand_prefix_score=np.full((B, c), np.nan), cand_matches=np.full((B, c), -1, np.int32),
        prefix_scores=np.full((B, n_models), np.nan),
        cand_pass=np.zeros((B, c), bool), cand_prefix_scores=np.full((B, c, n_models), np.nan),
        margin=np.full(B, np.inf), list_margin=np.full(B, np.inf), literal_margin=np.full(B, np.inf),
        next_id=np.full(B, -1, np.int32), next_score=np.full(B, np.nan))

    for b in range(B):
        s_sorted, j_sorted = kc.above(b)
        n_above = len(j_sorted)
        nc = min(c, n_above)
        cj, cs = j_sorted[:nc], s_sorted[:nc]
        res.n_above[b] = n_above
        res.n_cand[b] = nc
        res.cand_id[b, :nc] = cj
        res.cand_score[b, :nc] = cs
        served = None
        if nc:
            rr, m = lookahead(q_prefix_bits[b], q_ids[b], prefix_rows(cj), id_rows(cj), segs)
            ok = passes(rr, m, params, k, segs)
            rm = rr if segs else rr[:, None]          # [nc, models]
            r = rm[:, 0]                              # model 0: the reported prefix score
            res.cand_prefix_score[b, :nc] = r
            res.cand_matches[b, :nc] = m
            res.cand_pass[b, :nc] = ok
            res.cand_prefix_scores[b, :nc] = rm
            hits = np.nonzero(ok)[0]
            shown = int(hits[0]) if hits.size else 0
            if hits.size:
                served = int(hits[0])
                res.status[b] = HIT
                res.entry_id[b] = cj[served]
                res.key_score[b] = cs[served]
            else:
                res.status[b] = REJECT
            res.prefix_score[b] = r[shown]
            res.prefix_scores[b] = rm[shown]
            res.token_matches[b] = m[shown]
        if n_above > c:
            res.next_id[b], res.next_score[b] = j_sorted[c], s_sorted[c]   # the best entry just outside C_q

        # decision margin: the smallest score change that alters status or entry_id. A gap between two scores
        # closes when each moves by half of it, so the decision holds while every score moves by less than
        # half the margin.
        taus = [t for _, _, t in segs] if segs else [tau_a]

        def flip(r_row, m_val):
            # the smallest prefix-score change that flips a pass bit (none where the token ids decide it)
            if uses_r and (not uses_m or m_val >= tmin):
                return min(abs(r_row[h] - taus[h]) for h in range(len(taus)))
            return np.inf

        gaps = []
        if nc:
            for i in range((served if served is not None else nc - 1) + 1):   # candidates examined
                gaps.append(flip(rm[i], m[i]))
        if served is not None:
            gaps.append(cs[served] - tau_c)                         # j* falls out of A_q
            if n_above > c:
                # j* pushed past the cut: every entry ranked below it down to the one at the cut rises above it.
                # This also covers any single entry from past the cut overtaking j*.
                gaps.append(cs[served] - s_sorted[c])
            for i in range(nc):
                if i != served and ok[i]:
                    gaps.append(abs(cs[served] - cs[i]))            # another passing candidate overtakes j*
                elif i > served:                                    # a later failing one overtakes j* and passes
                    gaps.append(max(cs[served] - cs[i], flip(rm[i], m[i])))
        elif n_above < c:
            gaps.append(kc.closest[b])                              # any entry entering or leaving A_q
        else:
            gaps.append(cs[0] - tau_c)                              # every candidate leaving A_q
            gaps.append(cs[-1] - kc.below[b])                       # an entry from below tau_c entering C_q
            # entries past the cut rising above the last candidate: a passing one is served, a failing one only
            # if its pass bit flips too. Those farther below than the smallest gap so far cannot matter.
            bound = min(gaps)
            past = [i for i in range(c, n_above) if cs[-1] - s_sorted[i] < bound]
            if past:
                je = j_sorted[past]
                re, me = lookahead(q_prefix_bits[b], q_ids[b], prefix_rows(je), id_rows(je), segs)
                oke = passes(re, me, params, k, segs)
                rme = re if segs else re[:, None]
                for t, i in enumerate(past):
                    key = cs[-1] - s_sorted[i]
                    gaps.append(key if oke[t] else max(key, flip(rme[t], me[t])))
        res.margin[b] = min(gaps) if gaps else np.inf

        # candidate-list margin: the smallest score change that alters C_q or its order
        lgaps = [abs(x - tau_c) for x in cs]
        if n_above < c:
            lgaps.append(kc.closest[b])
        lgaps += [s_sorted[i] - s_sorted[i + 1] for i in range(min(c, n_above - 1))]
        res.list_margin[b] = min(lgaps) if lgaps else np.inf

        lit = [abs(kc.best[b] - tau_c)] if np.isfinite(kc.best[b]) else []
        if n_above >= 2:
            lit.append(s_sorted[0] - s_sorted[1])
        res.literal_margin[b] = min(lit) if lit else np.inf
    return res


def lookup(store: Store, queries: dict, params: Params, block_rows: int = 1 << 16) -> Result:
    """Algorithm 1's two checks for a batch, against every valid entry of a resident store.

    queries: {"emb": uint16 [B, d], "prefix": uint16 [B, d], "ids": int32 [B, k]} (bf16 bit patterns).
    """
    kc = KeyCheck(queries["emb"], params.tau_c)
    for j0 in range(0, store.n, block_rows):
        kc.add_rows(store.key[j0:min(store.n, j0 + block_rows)], j0)
    return decide(kc, queries["prefix"], queries["ids"], params,
                  lambda j: store.prefix[j], lambda j: store.ids[j])
