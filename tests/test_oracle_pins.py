"""Pins of the fp64 oracle against facts fixed by the paper or by mathematics (CPU only).

Each test is chosen so that a plausible slip in the oracle fails it. The slips covered are: a strict instead of
an inclusive threshold, the wrong tie order, serving the top candidate instead of the first passing one, scoring
the prefix against the key rows, set instead of positional token matching, a transposed operand, a dropped margin
term, and a wrong bf16 rounding.
"""
import json
import math
import os
import struct
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import CHECK_BOTH, CHECK_EMB, CHECK_TOKENS, HIT, MISS_KEY, REJECT, Params, Store

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bits(values):
    """bf16 bit patterns of values that are exactly representable in bf16 (checked)."""
    out = []
    for v in np.asarray(values, dtype=np.float64).ravel():
        u = struct.unpack("<I", struct.pack("<f", float(v)))[0]
        assert u & 0xFFFF == 0, f"{v} is not a bf16 value"
        assert struct.unpack("<f", struct.pack("<I", u))[0] == v
        out.append(u >> 16)
    return np.array(out, dtype=np.uint16).reshape(np.shape(values))


def exact(b):
    """Exact rational value of a bf16 bit pattern, from the IEEE-754 binary32 layout."""
    v = struct.unpack("<f", struct.pack("<I", int(b) << 16))[0]
    return Fraction(v)


def store_of(keys, prefixes, ids):
    return Store.of(bits(keys), bits(prefixes), np.asarray(ids, np.int32))


def queries_of(q, qp, qids):
    return {"emb": bits(np.atleast_2d(q)), "prefix": bits(np.atleast_2d(qp)),
            "ids": np.atleast_2d(np.asarray(qids, np.int32))}


E = np.eye(4)


# --- bf16 conversions ------------------------------------------------------------------------------------------

def test_widen_known_patterns():
    pats = np.array([0x3F80, 0xBF80, 0x3F00, 0x4049, 0x0001, 0x7F80, 0x0000, 0x8000], np.uint16)
    want = [1.0, -1.0, 0.5, 3.140625, 2.0 ** -133, math.inf, 0.0, -0.0]
    got = oracle.widen(pats)
    assert list(got) == want
    assert math.copysign(1.0, got[-1]) == -1.0


def test_round_to_bf16_ties_to_even():
    x = np.array([1.0, 1 + 2 ** -8, 1 + 3 * 2 ** -8, 1 + 2 ** -8 + 2 ** -20, -(1 + 2 ** -8), 3.4e38, 2.0 ** -130,
                  2.0 ** -140], np.float32)
    # 1+2^-8 is the midpoint of 1 (even) and 1+2^-7 (odd): stays 1. 1+3*2^-8 lies between 1+2^-7 (odd) and
    # 1+2^-6 (even): goes up. Just above a midpoint rounds up. 3.4e38 is past the largest bf16 (0x7F7F) and
    # rounds to inf. 2^-130 is a bf16 subnormal (fraction bit 3); 2^-140 is below half the smallest one, 2^-133.
    want = [0x3F80, 0x3F80, 0x3F82, 0x3F81, 0xBF80, 0x7F80, 0x0008, 0x0000]
    assert [int(v) for v in oracle.round_to_bf16(x)] == want


def test_round_to_bf16_keeps_nans_nan():
    # a NaN whose payload lies only in the dropped half would truncate to an infinity; it must stay a NaN of the
    # same sign (quieted: the top fraction bit set)
    x = np.array([0x7F800001, 0xFF800001, 0x7FC00000, 0x7FA00000], np.uint32).view(np.float32)
    got = [int(v) for v in oracle.round_to_bf16(x)]
    assert got == [0x7FC0, 0xFFC0, 0x7FC0, 0x7FE0]
    assert all(np.isnan(oracle.widen(np.array(got, np.uint16))))


def test_round_to_bf16_agrees_with_library():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.standard_normal(20000).astype(np.float32),
                        (rng.standard_normal(2000) * 1e-39).astype(np.float32),
                        np.array([np.inf, -np.inf, 0.0, -0.0, 65504.0, 1e38], np.float32)])
    lib = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.round_to_bf16(x), lib)


# --- stage 1 scores: closed forms ------------------------------------------------------------------------------

def test_scores_against_basis_vectors_are_the_query_components():
    # K = I: s_j = <q, e_j> = q_j exactly. A transposed operand or a row/column mix-up breaks this.
    q = np.array([0.5, -0.25, 0.75, 0.125])
    kc = oracle.KeyCheck(bits(q[None, :]), tau_c=-2.0)
    kc.add_rows(bits(E), 0)
    s, j = kc.above(0)
    assert list(j) == [2, 0, 3, 1]
    assert list(s) == [0.75, 0.5, 0.125, -0.25]


def test_scores_dyadic_closed_form():
    q = [0.5, 0.5, 0.5, 0.5]
    K = [[0.75, 0.25, -0.5, 0.125],      # 0.5 * 0.625 = 0.3125
         [1.0, 0.0, 0.0, 0.0],           # 0.5
         [-0.5, -0.5, -0.5, -0.5],       # -1
         [0.5, 0.5, 0.5, 0.5]]           # 1
    kc = oracle.KeyCheck(bits(np.array([q])), tau_c=-2.0)
    kc.add_rows(bits(np.array(K)), 100)
    s, j = kc.above(0)
    assert dict(zip(j.tolist(), s.tolist())) == {100: 0.3125, 101: 0.5, 102: -1.0, 103: 1.0}
    assert kc.best[0] == 1.0


# --- hand-built decisions --------------------------------------------------------------------------------------

def test_exact_duplicate_key_hits_lower_id():
    keys = [E[1], E[0], E[0], E[2]]
    pre = [E[3], E[1], E[1], E[2]]
    st = store_of(keys, pre, [[1, 2], [3, 4], [3, 4], [5, 6]])
    r = oracle.lookup(st, queries_of(E[0], E[1], [3, 4]), Params(0.9, 0.9, 4))
    assert r.status[0] == HIT and r.entry_id[0] == 1
    assert list(r.cand_id[0]) == [1, 2, -1, -1]
    assert r.key_score[0] == 1.0 and r.prefix_score[0] == 1.0 and r.token_matches[0] == 2


def test_first_passing_candidate_is_served_not_the_top_one():
    # entries 0 and 1 share the key; entry 0's prefix differs from the query's, entry 1's matches.
    st = store_of([E[0], E[0], E[1]], [E[2], E[3], E[3]], [[0, 0], [1, 1], [1, 1]])
    r = oracle.lookup(st, queries_of(E[0], E[3], [1, 1]), Params(0.5, 0.5, 3))
    assert r.status[0] == HIT and r.entry_id[0] == 1
    assert list(r.cand_id[0]) == [0, 1, -1]
    assert list(r.cand_prefix_score[0, :2]) == [0.0, 1.0]


def test_collision_with_distinct_prefix_is_rejected():
    # the threat model's key collision: same key, semantically distinct response prefix.
    st = store_of([E[0]], [E[1]], [[7, 8]])
    r = oracle.lookup(st, queries_of(E[0], E[2], [9, 9]), Params(0.85, 0.8, 4))
    assert r.status[0] == REJECT and r.entry_id[0] == -1
    assert r.n_cand[0] == 1 and r.prefix_score[0] == 0.0 and r.token_matches[0] == 0
    assert r.key_score[0] == 1.0


def test_reject_shows_the_first_candidate():
    # two candidates, neither passing: the shown lookahead score and token matches are those of the first (the
    # higher key score), not of the last
    st = store_of([E[0], [0.875, 0, 0, 0]], [[0.25, 0, 0, 0], [0.5, 0, 0, 0]], [[1, 2], [1, 0]])
    r = oracle.lookup(st, queries_of(E[0], E[0], [1, 2]), Params(0.5, 0.75, 4, check_mode=CHECK_BOTH))
    assert r.status[0] == REJECT and list(r.cand_id[0, :2]) == [0, 1]
    assert r.prefix_score[0] == 0.25 and r.token_matches[0] == 2
    assert list(r.cand_prefix_score[0, :2]) == [0.25, 0.5] and list(r.cand_matches[0, :2]) == [2, 1]


def test_prefix_check_reads_prefix_rows_not_key_rows():
    # key rows equal the query's prefix: scoring the prefix against key rows would wrongly pass.
    st = store_of([E[0]], [E[1]], [[0]])
    r = oracle.lookup(st, queries_of(E[0], E[0], [0]), Params(0.5, 0.5, 1))
    assert r.status[0] == REJECT


def test_all_below_threshold_is_a_key_miss():
    st = store_of([E[0], E[1]], [E[0], E[1]], [[0], [1]])
    q = np.array([0.5, 0.5, 0.5, 0.5])
    r = oracle.lookup(st, queries_of(q, q, [0]), Params(0.75, 0.0, 2))
    assert r.status[0] == MISS_KEY and r.n_cand[0] == 0 and r.entry_id[0] == -1
    assert r.key_score[0] == 0.5 and np.isnan(r.prefix_score[0]) and r.token_matches[0] == -1


def test_thresholds_are_inclusive():
    q = np.array([0.5, 0.5, 0.5, 0.5])
    st = store_of([E[0]], [E[0]], [[0]])
    qs = queries_of(q, q, [0])            # s = r = 0.5 exactly
    assert oracle.lookup(st, qs, Params(0.5, 0.5, 1)).status[0] == HIT
    assert oracle.lookup(st, qs, Params(np.nextafter(0.5, 1), 0.5, 1)).status[0] == MISS_KEY
    assert oracle.lookup(st, qs, Params(0.5, np.nextafter(0.5, 1), 1)).status[0] == REJECT


def test_top_c_cut_and_order():
    q = np.array([1.0, 0, 0, 0])
    keys = [[0.5, 0.5, 0.5, 0.5], [0.75, 0, 0, 0], [1.0, 0, 0, 0], [0.875, 0, 0, 0], [0.25, 0, 0, 0]]
    st = store_of(keys, [E[1]] * 5, [[0]] * 5)
    r = oracle.lookup(st, queries_of(q, E[2], [1]), Params(0.4, 0.9, 3))
    assert list(r.cand_id[0]) == [2, 3, 1]
    assert list(r.cand_score[0]) == [1.0, 0.875, 0.75]
    assert r.n_above[0] == 4 and r.n_cand[0] == 3 and r.status[0] == REJECT


def test_token_matches_are_positional():
    st = store_of([E[0]], [E[1]], [[1, 2, 3, 4]])
    r = oracle.lookup(st, queries_of(E[0], E[1], [4, 3, 2, 1]), Params(0.5, 0.5, 1))
    assert r.token_matches[0] == 0           # same multiset, no position equal
    r = oracle.lookup(st, queries_of(E[0], E[1], [1, 9, 3, 9]), Params(0.5, 0.5, 1))
    assert r.token_matches[0] == 2


def test_check_modes():
    st = store_of([E[0], E[0]], [E[1], E[2]], [[1, 2, 3], [1, 2, 9]])
    qs = queries_of(E[0], E[2], [1, 2, 3])   # entry 0: ids equal, prefix orthogonal; entry 1: prefix equal
    tok = oracle.lookup(st, qs, Params(0.5, 0.5, 2, CHECK_TOKENS))             # Algorithm 1: all k equal
    assert tok.status[0] == HIT and tok.entry_id[0] == 0
    emb = oracle.lookup(st, qs, Params(0.5, 0.5, 2, CHECK_EMB))
    assert emb.status[0] == HIT and emb.entry_id[0] == 1
    both = oracle.lookup(st, qs, Params(0.5, 0.5, 2, CHECK_BOTH))
    assert both.status[0] == REJECT
    loose = oracle.lookup(st, qs, Params(0.5, 0.5, 2, CHECK_BOTH, token_match_min=2))
    assert loose.status[0] == HIT and loose.entry_id[0] == 1


def test_empty_cache():
    st = Store.of(np.zeros((0, 4), np.uint16), np.zeros((0, 4), np.uint16), np.zeros((0, 2), np.int32))
    r = oracle.lookup(st, queries_of(E[0], E[0], [0, 0]), Params(0.5, 0.5, 2))
    assert r.status[0] == MISS_KEY and r.key_score[0] == -np.inf and r.margin[0] == np.inf


# --- margin -----------------------------------------------------------------------------------------------------

def test_margin_terms():
    q = np.array([1.0, 0, 0, 0])
    # two passing candidates 2^-8 apart in key score: the served one could flip.
    st = store_of([[1.0, 0, 0, 0], [0.99609375, 0, 0, 0]], [E[1], E[1]], [[0], [0]])
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.5, 0.5, 2))
    assert r.entry_id[0] == 0 and r.margin[0] == 1.0 - 0.99609375
    # the only candidate's prefix score sits 2^-6 above tau_a: the lookahead margin.
    st = store_of([E[0]], [[0.5, 0.5, 0.5, 0.5]], [[0]])
    r = oracle.lookup(st, queries_of(q, [0.5, 0.5, 0.5, 0.5], [0]), Params(0.25, 0.984375, 1))
    assert r.status[0] == HIT and r.margin[0] == 1.0 - 0.984375
    # fewer candidates than c and nothing served: the closest score to tau_c anywhere counts (entry 1, 0.5).
    st = store_of([E[0], [0.5, 0.5, 0.5, 0.5]], [E[2], E[2]], [[0], [0]])
    r = oracle.lookup(st, queries_of(q, E[3], [0]), Params(0.53125, 0.5, 4))
    assert r.status[0] == REJECT and r.margin[0] == 0.03125
    # more candidates than c, all failing: the cut between candidates 2 and 3 (2^-6) reorders the list but
    # cannot change the decision unless the entry past the cut would pass.
    keys = [E[0], [0.875, 0, 0, 0], [0.859375, 0, 0, 0]]
    st = store_of(keys, [E[2]] * 3, [[0]] * 3)
    r = oracle.lookup(st, queries_of(q, E[3], [0]), Params(0.5, 0.5, 2))
    assert r.status[0] == REJECT and r.margin[0] == 0.5
    assert r.list_margin[0] == 0.875 - 0.859375 and r.next_id[0] == 2 and r.next_score[0] == 0.859375
    st = store_of(keys, [E[2], E[2], E[3]], [[0]] * 3)
    r = oracle.lookup(st, queries_of(q, E[3], [0]), Params(0.5, 0.5, 2))
    assert r.status[0] == REJECT and r.margin[0] == 0.875 - 0.859375
    # the served entry is the last candidate: being pushed past the cut would change the decision.
    st = store_of(keys, [E[2], E[3], E[3]], [[0]] * 3)
    r = oracle.lookup(st, queries_of(q, E[3], [0]), Params(0.5, 0.5, 2))
    assert r.status[0] == HIT and r.entry_id[0] == 1 and r.margin[0] == 0.875 - 0.859375
    # the served entry's key score sits 2^-6 above tau_c, its prefix score 0.5 above tau_a: falling out of A_q is
    # the closest change.
    st = store_of([E[0]], [E[1]], [[0]])
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.984375, 0.5, 1))
    assert r.status[0] == HIT and r.margin[0] == 1.0 - 0.984375


def test_literal_margin_is_the_threshold_distance_or_the_top_two_gap():
    """The north-star's literal band: min(|best score - tau_c|, s_(1) - s_(2)), from dyadic scores."""
    q = np.array([1.0, 0, 0, 0])
    keys = [[0.875, 0, 0, 0], [0.75, 0, 0, 0], [0.5, 0, 0, 0]]
    st = store_of(keys, [E[1]] * 3, [[0]] * 3)
    # best 0.875 is 0.125 above tau_c = 0.75; the top two (0.875, 0.75) are 0.125 apart: both terms 0.125
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.75, 0.5, 2))
    assert r.literal_margin[0] == 0.125
    # tau_c = 0.8125: the best is 0.0625 above it; only one entry clears it, so no top-two gap
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.8125, 0.5, 2))
    assert r.n_above[0] == 1 and r.literal_margin[0] == 0.0625
    # tau_c = 0.25: the best is 0.625 above it, and the top-two gap 0.125 is smaller
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.25, 0.5, 3))
    assert r.literal_margin[0] == 0.125
    # nothing clears tau_c = 0.9375: the distance of the best score (0.875) below it
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.9375, 0.5, 2))
    assert r.status[0] == MISS_KEY and r.literal_margin[0] == 0.0625
    # an empty cache has no score at all: no band
    empty = Store.of(np.zeros((0, 4), np.uint16), np.zeros((0, 4), np.uint16), np.zeros((0, 1), np.int32))
    r = oracle.lookup(empty, queries_of(q, E[1], [0]), Params(0.5, 0.5, 2))
    assert r.literal_margin[0] == math.inf


def test_margin_counts_changes_from_outside_the_examined_candidates():
    q = np.array([1.0, 0, 0, 0])
    # a passing entry just past the cut could rise above the served entry and be served instead
    keys = [E[0], [0.99609375, 0, 0, 0], [0.9921875, 0, 0, 0]]
    st = store_of(keys, [E[1], E[2], E[1]], [[0]] * 3)
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.5, 0.5, 2))
    assert r.status[0] == HIT and r.entry_id[0] == 0 and r.margin[0] == 1.0 - 0.9921875
    # a failing candidate after the served one, 2^-8 below it in key score and 2^-8 short of tau_a
    st = store_of(keys[:2], [E[1], [0, 0.49609375, 0, 0]], [[0]] * 2)
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.5, 0.5, 2))
    assert r.status[0] == HIT and r.entry_id[0] == 0 and r.margin[0] == 0.5 - 0.49609375
    # a full candidate list rejected, and a passing entry 2^-8 below tau_c that could overtake the last candidate
    keys = [E[0], [0.50390625, 0, 0, 0], [0.49609375, 0, 0, 0]]
    st = store_of(keys, [E[2], E[2], E[1]], [[0]] * 3)
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.5, 0.5, 2))
    assert r.status[0] == REJECT and r.margin[0] == 0.50390625 - 0.49609375
    # rejected, the entry at the cut fails, and the one after it passes
    keys = [E[0], [0.99609375, 0, 0, 0], [0.9921875, 0, 0, 0]]
    st = store_of(keys, [E[2], E[2], E[1]], [[0]] * 3)
    r = oracle.lookup(st, queries_of(q, E[1], [0]), Params(0.5, 0.5, 1))
    assert r.status[0] == REJECT and r.margin[0] == 1.0 - 0.9921875


def _decision_from_scores(s, r, m, tau_c, taus, c, mode, tmin):
    """Algorithm 1's decision for one query from its key scores s[j], prefix scores r[j][h] and token matches m[j]."""
    above = sorted((j for j in range(len(s)) if s[j] >= tau_c), key=lambda j: (-s[j], j))
    for j in above[:c]:
        emb = all(r[j][h] >= taus[h] for h in range(len(taus)))
        tok = m[j] >= tmin
        if (emb if mode == CHECK_EMB else tok if mode == CHECK_TOKENS else emb and tok):
            return HIT, j
    return (REJECT if above else MISS_KEY), -1


@pytest.mark.parametrize("seed", range(40))
def test_decision_survives_every_score_change_below_half_the_margin(seed):
    """The margin's defining property: moving every key and prefix score by less than half the decision margin
    (so that no gap between two scores closes) leaves the status and the served entry unchanged. Scores sit on a
    2^-8 grid around the thresholds, so ties, near ties and entries on both sides of the cut are common."""
    rng = np.random.default_rng(1000 + seed)
    step, tau_c = 2.0 ** -8, 0.75
    models = 2 if seed % 4 == 3 else 1
    taus = [0.625, 0.5625][:models]
    mode = [CHECK_EMB, CHECK_EMB, CHECK_TOKENS, CHECK_BOTH][seed % 4] if models == 1 else CHECK_EMB
    for _ in range(25):
        n, c, kt = int(rng.integers(1, 11)), int(rng.integers(1, 5)), 3
        s = tau_c + step * rng.integers(-12, 13, size=n)
        s[rng.random(n) < 0.15] = 0.5
        rv = np.array(taus)[None, :] + step * rng.integers(-12, 13, size=(n, models))
        keys = np.zeros((n, 4))
        keys[:, 0] = s
        pre = np.zeros((n, 2 * models))
        pre[:, 0::2] = rv
        ids = rng.integers(0, 2, size=(n, kt))
        qi = rng.integers(0, 2, size=kt)
        tmin = int(rng.integers(1, kt + 1))
        qp = np.tile([1.0, 0.0], models)
        p = Params(tau_c, taus[0], c, check_mode=mode, token_match_min=tmin,
                   prefix_dims=(2,) * models if models > 1 else None,
                   tau_a_models=tuple(taus) if models > 1 else None)
        res = oracle.lookup(store_of(keys, pre, ids), queries_of(E[0], qp, qi), p)
        m = (ids == qi[None, :]).sum(axis=1)
        got = (int(res.status[0]), int(res.entry_id[0]))
        assert _decision_from_scores(s, rv, m, tau_c, taus, c, mode, tmin) == got
        mu = float(res.margin[0])
        if mu == 0.0:
            continue
        delta = 0.49 * min(mu, 1.0)
        moves = [(rng.uniform(-delta, delta, n), rng.uniform(-delta, delta, (n, models))) for _ in range(60)]
        moves += [(delta * rng.choice([-1.0, 1.0], n), delta * rng.choice([-1.0, 1.0], (n, models)))
                  for _ in range(60)]
        for e in range(n):                 # one entry moves one way, every other entry the other way
            for ss in (-1.0, 1.0):
                for sr in (-1.0, 1.0):
                    ds, dr = np.full(n, -ss * delta), np.full((n, models), -sr * delta)
                    ds[e], dr[e] = ss * delta, sr * delta
                    moves.append((ds, dr))
        for ds, dr in moves:
            assert _decision_from_scores(s + ds, rv + dr, m, tau_c, taus, c, mode, tmin) == got, \
                f"margin {mu}: scores {s}, prefix scores {rv.tolist()}, c {c}, moved by {ds}, {dr.tolist()}"


# --- brute force in exact arithmetic on tiny inputs ---------------------------------------------------------------

def _brute(keys_b, pre_b, ids, q_b, p_b, t, tau_c, tau_a, c):
    """Exact rational scores; candidates by repeated selection of the best remaining entry."""
    n = len(keys_b)
    s = [sum(exact(a) * exact(b) for a, b in zip(q_b, keys_b[j])) for j in range(n)]
    remaining = [j for j in range(n) if s[j] >= Fraction(tau_c)]
    cand = []
    while remaining and len(cand) < c:
        best = remaining[0]
        for j in remaining[1:]:
            if s[j] > s[best]:          # equal scores keep the earlier (lower) id
                best = j
        cand.append(best)
        remaining.remove(best)
    r = [sum(exact(a) * exact(b) for a, b in zip(p_b, pre_b[j])) for j in cand]
    served = next((i for i, j in enumerate(cand) if r[i] >= Fraction(tau_a)), None)
    return s, cand, r, served


@pytest.mark.parametrize("seed", range(12))
def test_brute_force_exact_arithmetic(seed):
    rng = np.random.default_rng(seed)
    n, d, k, B, c = int(rng.integers(1, 13)), int(rng.integers(1, 9)), 3, 4, int(rng.integers(1, 5))
    grid = np.arange(-8, 9) / 8.0                        # dyadic values: exact in bf16
    keys = rng.choice(grid, size=(n, d))
    keys[rng.integers(0, n)] = keys[0]                    # force a duplicate key
    pre = rng.choice(grid, size=(n, d))
    ids = rng.integers(0, 3, size=(n, k))
    qs = rng.choice(grid, size=(B, d))
    qs[0] = keys[0]
    qp = rng.choice(grid, size=(B, d))
    qp[0] = pre[0]
    qi = rng.integers(0, 3, size=(B, k))
    tau_c, tau_a = float(rng.choice([-0.5, 0.0, 0.25])), float(rng.choice([0.0, 0.5]))
    res = oracle.lookup(store_of(keys, pre, ids), queries_of(qs, qp, qi), Params(tau_c, tau_a, c))
    kb, pb = bits(keys), bits(pre)
    for b in range(B):
        s, cand, r, served = _brute(kb, pb, ids, bits(qs[b]), bits(qp[b]), qi[b], tau_c, tau_a, c)
        assert list(res.cand_id[b, :len(cand)]) == cand and res.n_cand[b] == len(cand)
        for i, j in enumerate(cand):
            assert res.cand_score[b, i] == float(s[j])        # exact: fp64 holds these sums exactly
            assert res.cand_prefix_score[b, i] == float(r[i])
        if served is None:
            assert res.status[b] == (REJECT if cand else MISS_KEY) and res.entry_id[b] == -1
        else:
            assert res.status[b] == HIT and res.entry_id[b] == cand[served]
        assert res.key_score[b] == (float(s[cand[served]]) if served is not None else float(max(s)))


# --- special cases that reduce to library routines ----------------------------------------------------------------

def _random_unit_bits(rng, n, d):
    x = rng.standard_normal((n, d))
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    return oracle.round_to_bf16(x.astype(np.float32))


def test_top1_with_open_thresholds_is_maximum_inner_product_search():
    rng = np.random.default_rng(7)
    K = _random_unit_bits(rng, 300, 16)
    K[200] = K[17]                                       # an exact tie: the lower id must win
    Q = np.concatenate([_random_unit_bits(rng, 20, 16), K[17:18]])
    st = Store.of(K, K, np.zeros((300, 1), np.int32))
    res = oracle.lookup(st, {"emb": Q, "prefix": Q, "ids": np.zeros((21, 1), np.int32)}, Params(-2.0, -2.0, 1))
    kf = oracle.widen(K)
    for b in range(21):
        scores = [math.fsum(x * y for x, y in zip(oracle.widen(Q[b]), kf[j])) for j in range(300)]
        assert res.entry_id[b] == int(np.argmax(scores))  # numpy argmax returns the first maximum
    assert res.entry_id[20] == 17


def test_open_threshold_with_c_equal_n_is_a_stable_sort():
    rng = np.random.default_rng(8)
    K = _random_unit_bits(rng, 64, 8)
    K[40] = K[3]
    K[41] = K[3]
    Q = K[3:4].copy()
    st = Store.of(K, K, np.zeros((64, 1), np.int32))
    res = oracle.lookup(st, {"emb": Q, "prefix": Q, "ids": np.zeros((1, 1), np.int32)}, Params(-2.0, 2.0, 64))
    kf, qf = oracle.widen(K), oracle.widen(Q[0])
    scores = np.array([math.fsum(x * y for x, y in zip(qf, kf[j])) for j in range(64)])
    assert list(res.cand_id[0]) == list(np.argsort(-scores, kind="stable"))
    assert list(res.cand_id[0, :3]) == [3, 40, 41]


# --- invariants on clustered random inputs -------------------------------------------------------------------------

def test_invariants_and_query_order_independence():
    rng = np.random.default_rng(11)
    n, d, k, B, c = 500, 32, 4, 40, 5
    cent = rng.standard_normal((10, d))
    keys = cent[rng.integers(0, 10, n)] + 0.15 / math.sqrt(d) * rng.standard_normal((n, d))
    keys /= np.linalg.norm(keys, axis=1, keepdims=True)
    K = oracle.round_to_bf16(keys.astype(np.float32))
    P = _random_unit_bits(rng, n, d)
    T = rng.integers(0, 5, (n, k)).astype(np.int32)
    tgt = rng.integers(0, n, B)
    qf = keys[tgt] + 0.05 / math.sqrt(d) * rng.standard_normal((B, d))
    Q = oracle.round_to_bf16((qf / np.linalg.norm(qf, axis=1, keepdims=True)).astype(np.float32))
    QP = P[tgt].copy()
    QP[::3] = _random_unit_bits(rng, len(QP[::3]), d)
    QT = T[tgt].copy()
    params = Params(0.9, 0.8, c)
    st = Store.of(K, P, T)
    res = oracle.lookup(st, {"emb": Q, "prefix": QP, "ids": QT}, params)
    assert np.all(np.abs(res.cand_score[res.cand_id >= 0]) <= 1 + 1e-2)
    assert np.all(res.n_cand == np.minimum(c, res.n_above))
    for b in range(B):
        nc = res.n_cand[b]
        cs, cj = res.cand_score[b, :nc], res.cand_id[b, :nc]
        assert np.all(cs >= params.tau_c)
        assert all((cs[i] > cs[i + 1]) or (cs[i] == cs[i + 1] and cj[i] < cj[i + 1]) for i in range(nc - 1))
        if res.status[b] == HIT:
            assert res.entry_id[b] in cj
            assert res.key_score[b] >= params.tau_c and res.prefix_score[b] >= params.tau_a
        else:
            assert res.entry_id[b] == -1
    assert np.sum(res.status == HIT) > 10 and np.sum(res.status == REJECT) > 5
    perm = rng.permutation(B)
    res2 = oracle.lookup(st, {"emb": Q[perm], "prefix": QP[perm], "ids": QT[perm]}, params)
    assert np.array_equal(res2.entry_id, res.entry_id[perm]) and np.array_equal(res2.status, res.status[perm])
    assert np.array_equal(res2.cand_id, res.cand_id[perm])
    # the store read block by block gives the same A_q as one pass
    res3 = oracle.lookup(st, {"emb": Q, "prefix": QP, "ids": QT}, params, block_rows=7)
    assert np.array_equal(res3.cand_id, res.cand_id) and np.array_equal(res3.margin, res.margin)


# --- the paper's printed counts ---------------------------------------------------------------------------------------

def test_table3_end_to_end_is_key_and_lookahead():
    """Table 3: end-to-end passes are exactly the cache-check passes that also pass the lookahead check."""
    with open(os.path.join(GOLDEN, "table3_adaptive.json")) as f:
        table = json.load(f)
    d = 64
    for row in table["rows"]:
        n, key_pass, la_pass = row["queries"], row["cache_check"], row["lookahead_given_cache"]
        # entry i is the victim of query i; the first `cache_check` queries carry its key, the first
        # `lookahead_given_cache` of those also its response prefix.
        rng = np.random.default_rng(n + key_pass)
        keys = _random_unit_bits(rng, n, d)
        pre = _random_unit_bits(rng, n, d)
        ids = rng.integers(0, 100, (n, 4)).astype(np.int32)
        q = np.zeros((n, d), np.uint16)
        qp = np.zeros((n, d), np.uint16)
        for i in range(n):
            q[i] = keys[i] if i < key_pass else _random_unit_bits(rng, 1, d)[0]
            qp[i] = pre[i] if i < la_pass else _random_unit_bits(rng, 1, d)[0]
        st = Store.of(keys, pre, ids)
        # At d = 64 random unit vectors have cosine ~N(0, 1/64), far below 0.9, while an exact copy of a
        # bf16-rounded unit vector scores 1 +- 2^-8: only the planted matches clear either threshold.
        res = oracle.lookup(st, {"emb": q, "prefix": qp, "ids": ids}, Params(0.9, 0.9, 1))
        key_hits = int(np.sum(res.status != MISS_KEY))
        e2e = int(np.sum(res.status == HIT))
        assert key_hits == row["cache_check"]
        assert e2e == row["lookahead_given_cache"] == row["end_to_end"]
        assert np.all(res.entry_id[res.status == HIT] == np.nonzero(res.status == HIT)[0])


# --- serve loop -----------------------------------------------------------------------------------------------------

def test_serve_loop_appends_misses_in_query_order():
    params = Params(0.9, 0.9, 2)
    loop = oracle.ServeLoop(16, 4, 2, params)
    loop.insert(bits([E[0]]), bits([E[0]]), np.array([[0, 0]], np.int32))
    # victim x = e1 with response prefix e1; the adversary's x* = e1 with a different response prefix e2.
    adv = queries_of(E[1], E[2], [6, 6])
    r, first, m = loop.step(adv)
    assert r.status[0] == MISS_KEY and (first, m) == (1, 1)
    victim = queries_of(np.array([E[1], E[0]]), np.array([E[1], E[0]]), [[5, 5], [0, 0]])
    r, first, m = loop.step(victim)
    # the victim collides with x*'s entry but its own prefix differs: rejected, decoded and appended.
    assert list(r.status) == [REJECT, HIT] and r.entry_id[1] == 0
    assert (first, m) == (2, 1)
    assert np.array_equal(loop.store.key[2], bits(E[1])) and list(loop.store.ids[2]) == [5, 5]
    # a later paraphrase of the victim sees x*'s entry first (lower id), which fails, then the victim's.
    r, first, m = loop.step(queries_of(E[1], E[1], [5, 5]))
    assert r.status[0] == HIT and r.entry_id[0] == 2 and list(r.cand_id[0]) == [1, 2] and m == 0
