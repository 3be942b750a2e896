"""Pins of the oracle's ensemble of m lookahead checks (section 3.4, "Analysis"; Figure 6).

A hit is valid only if the key check holds and every one of the m lookahead checks holds, each with its own
embedding model and threshold. The paper's claim is that m checks that each pass an attack with probability at
most p2 detect it with probability at least 1 - p2^m. These tests pin the conjunction, the per-model
thresholds and the reduction to one check.
"""
import numpy as np
import pytest

import oracle
from oracle import HIT, REJECT, Params, Store

from test_oracle_pins import bits, queries_of, store_of

E = np.eye(4)


def _ens(*dims_taus):
    dims = tuple(d for d, _ in dims_taus)
    taus = tuple(t for _, t in dims_taus)
    return dims, taus


def test_every_model_must_pass():
    # one entry; the prefix row is two 4-dim model segments
    key = [E[0]]
    pre = [np.concatenate([E[1], E[2]])]
    st = store_of(key, pre, [[0]])
    dims, taus = _ens((4, 0.5), (4, 0.5))
    p = Params(0.5, 0.0, 1, prefix_dims=dims, tau_a_models=taus)
    both = oracle.lookup(st, queries_of(E[0], np.concatenate([E[1], E[2]]), [0]), p)
    assert both.status[0] == HIT and list(both.prefix_scores[0]) == [1.0, 1.0]
    first_only = oracle.lookup(st, queries_of(E[0], np.concatenate([E[1], E[3]]), [0]), p)
    assert first_only.status[0] == REJECT and list(first_only.prefix_scores[0]) == [1.0, 0.0]
    second_only = oracle.lookup(st, queries_of(E[0], np.concatenate([E[3], E[2]]), [0]), p)
    assert second_only.status[0] == REJECT and second_only.prefix_score[0] == 0.0


def test_each_model_uses_its_own_threshold():
    half = np.array([0.75, 0.5, 0.25, 0.0])          # <half, e0> = 0.75 exactly
    st = store_of([E[0]], [np.concatenate([E[0], E[0]])], [[0]])
    q = queries_of(E[0], np.concatenate([half, half]), [0])
    for taus, want in [((0.7, 0.7), HIT), ((0.7, 0.8), REJECT), ((0.8, 0.7), REJECT), ((0.75, 0.75), HIT)]:
        p = Params(0.5, 0.0, 1, prefix_dims=(4, 4), tau_a_models=taus)
        assert oracle.lookup(st, q, p).status[0] == want, taus


def test_thresholds_belong_to_their_models():
    # model 0 scores 0.75 and model 1 scores 0.5, so swapping the two thresholds changes the outcome
    a = np.array([0.75, 0.5, 0.25, 0.0])
    b = np.array([0.5, 0.5, 0.5, 0.5])
    st = store_of([E[0]], [np.concatenate([E[0], E[0]])], [[0]])
    q = queries_of(E[0], np.concatenate([a, b]), [0])
    for taus, want in [((0.7, 0.4), HIT), ((0.4, 0.7), REJECT), ((0.75, 0.5), HIT), ((0.5, 0.75), REJECT)]:
        r = oracle.lookup(st, q, Params(0.5, 0.0, 1, prefix_dims=(4, 4), tau_a_models=taus))
        assert r.status[0] == want, taus
        assert list(r.prefix_scores[0]) == [0.75, 0.5] and list(r.cand_prefix_scores[0, 0]) == [0.75, 0.5]


def test_single_model_ensemble_is_the_plain_check():
    rng = np.random.default_rng(5)
    n, d, B = 200, 16, 30
    x = rng.standard_normal((n, d))
    K = oracle.round_to_bf16((x / np.linalg.norm(x, axis=1, keepdims=True)).astype(np.float32))
    y = rng.standard_normal((n, d))
    P = oracle.round_to_bf16((y / np.linalg.norm(y, axis=1, keepdims=True)).astype(np.float32))
    T = rng.integers(0, 4, (n, 3)).astype(np.int32)
    idx = rng.integers(0, n, B)
    qs = {"emb": K[idx], "prefix": P[idx].copy(), "ids": T[idx]}
    qs["prefix"][::2] = P[rng.integers(0, n, len(qs["prefix"][::2]))]
    st = Store.of(K, P, T)
    plain = oracle.lookup(st, qs, Params(0.3, 0.5, 4))
    one = oracle.lookup(st, qs, Params(0.3, 0.0, 4, prefix_dims=(d,), tau_a_models=(0.5,)))
    for f in ("status", "entry_id", "cand_id", "cand_prefix_score", "margin"):
        assert np.array_equal(getattr(plain, f), getattr(one, f), equal_nan=True), f


@pytest.mark.parametrize("m", [1, 2, 3, 4])
def test_attack_pass_rate_falls_as_p_to_the_m(m):
    """Section 3.4: with m independent checks that each let an attack through with probability p, the attack
    passes them all with probability p^m (detection at least 1 - p^m)."""
    rng = np.random.default_rng(100 + m)
    n_adv, d, p_pass = 3000, 8, 0.5
    dims = tuple([d] * m)
    # entry j is the victim of query j: same key (the collision), and per model a prefix that either matches
    # the victim's (this model lets the attack through) or is orthogonal to it, independently with probability p
    keys = np.tile(E[0], (n_adv, 2))[:, :d]
    pres = np.tile(np.concatenate([np.eye(d)[1]] * m), (n_adv, 1))
    qpre = pres.copy()
    through = rng.random((n_adv, m)) < p_pass
    for h in range(m):
        qpre[~through[:, h], h * d:(h + 1) * d] = np.eye(d)[2]
    st = Store.of(bits(keys), bits(pres), np.zeros((n_adv, 1), np.int32))
    qs = {"emb": bits(keys), "prefix": bits(qpre), "ids": np.zeros((n_adv, 1), np.int32)}
    # every entry shares the key, so each query's candidates are entries 0..c-1; use c = 1 and a store of the
    # single victim row per query by giving each query its own one-entry store
    hits = 0
    for j in range(n_adv):
        one = Store.of(st.key[j:j + 1], st.prefix[j:j + 1], st.ids[j:j + 1])
        r = oracle.lookup(one, {"emb": qs["emb"][j:j + 1], "prefix": qs["prefix"][j:j + 1],
                                "ids": qs["ids"][j:j + 1]},
                          Params(0.9, 0.0, 1, prefix_dims=dims, tau_a_models=(0.5,) * m))
        hits += int(r.status[0] == HIT)
    rate = hits / n_adv
    want = p_pass ** m
    assert hits == int(np.sum(np.all(through, axis=1)))
    assert abs(rate - want) < 5 * np.sqrt(want * (1 - want) / n_adv)
