"""Pins of the oracle's SimHash index (Eq. 1; Algorithm 1's "search semantic cache with key h(x)").

The index's collision probability per bit is 1 - theta/pi for an angle theta (the published property of
random-hyperplane hashing). A Hamming radius over b bits then admits a pair at angle theta with the binomial
probability P[Binomial(b, theta/pi) <= radius], which gives the gapped-LSH property of Eq. 1.
"""
import math

import numpy as np
import pytest

import oracle
from oracle import Params, Store
from paper_2608_01718_gb300 import workloads as wl

from test_oracle_pins import bits


def _pair_at_angle(theta, d=64):
    x = np.zeros((1, d), np.float32)
    y = np.zeros((1, d), np.float32)
    x[0, 0] = 1.0
    y[0, 0], y[0, 1] = math.cos(theta), math.sin(theta)
    xb, yb = oracle.round_to_bf16(x), oracle.round_to_bf16(y)
    xf, yf = oracle.widen(xb)[0], oracle.widen(yb)[0]
    actual = math.acos(float(xf @ yf / np.linalg.norm(xf) / np.linalg.norm(yf)))
    return xb, yb, actual


@pytest.mark.parametrize("theta", [0.1, 0.5, 1.0, math.pi / 2, 2.5])
def test_bit_agreement_is_one_minus_theta_over_pi(theta):
    b = 8192
    R = wl.bf16_bits(wl.hyperplanes(b, 64, seed=int(theta * 1000)))
    xb, yb, actual = _pair_at_angle(theta)
    sx, _ = oracle.signatures(xb, R)
    sy, _ = oracle.signatures(yb, R)
    agree = float(np.mean(sx == sy))
    p = 1 - actual / math.pi
    assert abs(agree - p) < 5 * math.sqrt(p * (1 - p) / b) + 1e-9


def test_admitted_fraction_is_the_binomial_tail():
    scipy_stats = pytest.importorskip("scipy.stats")
    b, radius, trials = 64, 12, 4000
    xb, yb, actual = _pair_at_angle(0.5)
    admitted = 0
    for t in range(trials // 100):
        R = wl.bf16_bits(wl.hyperplanes(b * 100, 64, seed=t)).reshape(100, b, 64)
        for r in R:
            sx, _ = oracle.signatures(xb, r)
            sy, _ = oracle.signatures(yb, r)
            admitted += int(oracle.hamming(sx, sy)[0, 0] <= radius)
    want = scipy_stats.binom.cdf(radius, b, actual / math.pi)
    assert abs(admitted / trials - want) < 5 * math.sqrt(want * (1 - want) / trials)


def test_zero_projection_sets_the_bit_and_hamming_brute_force():
    R = bits(np.array([[1.0, 0, 0, 0], [0, 1.0, 0, 0], [0, 0, -1.0, 0]]))
    z = bits(np.array([[0.0, 0.5, 0.5, 0.5], [-0.5, -0.5, 0.5, 0.0]]))
    sig, amb = oracle.signatures(z, R)
    assert sig.tolist() == [[True, True, False], [False, False, False]]
    assert amb.tolist() == [[True, False, False], [False, False, False]]
    rng = np.random.default_rng(1)
    a, c = rng.random((7, 40)) < 0.5, rng.random((5, 40)) < 0.5
    brute = [[sum(int(u) ^ int(v) for u, v in zip(x, y)) for y in c] for x in a]
    assert oracle.hamming(a, c).tolist() == brute


def _small_case(seed=3, n=400, d=32, B=24):
    rng = np.random.default_rng(seed)
    cent = rng.standard_normal((8, d))
    cent /= np.linalg.norm(cent, axis=1, keepdims=True)
    keys = cent[rng.integers(0, 8, n)] + 0.15 / math.sqrt(d) * rng.standard_normal((n, d))
    keys /= np.linalg.norm(keys, axis=1, keepdims=True)
    K = oracle.round_to_bf16(keys.astype(np.float32))
    P = oracle.round_to_bf16(rng.standard_normal((n, d)).astype(np.float32) / math.sqrt(d))
    T = rng.integers(0, 4, (n, 3)).astype(np.int32)
    tgt = rng.integers(0, n, B)
    q = keys[tgt] + 0.05 / math.sqrt(d) * rng.standard_normal((B, d))
    q /= np.linalg.norm(q, axis=1, keepdims=True)
    Q = oracle.round_to_bf16(q.astype(np.float32))
    return Store.of(K, P, T), {"emb": Q, "prefix": P[tgt], "ids": T[tgt]}


def test_radius_at_least_b_is_the_exact_lookup():
    st, qs = _small_case()
    R = wl.bf16_bits(wl.hyperplanes(64, 32))
    p = Params(0.9, 0.5, 4)
    exact = oracle.lookup(st, qs, p)
    lsh, amb = oracle.lookup_lsh(st, qs, p, R, radius=64)
    assert not amb.any()
    for f in ("status", "entry_id", "cand_id", "n_cand", "margin"):
        assert np.array_equal(getattr(exact, f), getattr(lsh, f), equal_nan=True), f


def test_block_wise_check_is_the_whole_store_check():
    # the store through the SimHash key check in blocks of 7 rows (the last one ragged) gives the result of one
    # block: A_q is a union over blocks, and each block's ids are offset by its first row
    st, qs = _small_case()
    R = wl.bf16_bits(wl.hyperplanes(64, 32))
    p = Params(0.9, 0.5, 8)
    whole, amb1 = oracle.lookup_lsh(st, qs, p, R, radius=20)
    blocks, amb2 = oracle.lookup_lsh(st, qs, p, R, radius=20, block_rows=7)
    assert np.array_equal(amb1, amb2)
    for f in ("status", "entry_id", "cand_id", "cand_score", "n_cand", "n_above", "margin"):
        assert np.array_equal(getattr(whole, f), getattr(blocks, f), equal_nan=True), f
    assert np.any(whole.n_cand > 0)


def test_an_ambiguous_bit_at_the_radius_marks_the_query():
    # query 0's projection on hyperplane 0 is exactly zero (an ambiguous bit); entry 0 clears the key threshold and
    # differs from it in that bit only, so at radius 0 the entry's admission hangs on that bit and the query is
    # marked. Query 1 has no zero projection and an identical entry: not marked.
    d = 8
    R = np.zeros((4, d), np.float32)
    R[np.arange(4), np.arange(4)] = 1.0
    q = np.zeros((2, d), np.float32)
    q[0, 1:5] = 0.5
    q[1, 0:4] = 0.5
    k = np.zeros((2, d), np.float32)
    k[0, 0], k[0, 1:5] = -0.25, 0.5        # <q0, k0> = 1, sign differs on hyperplane 0 only
    k[1] = q[1]
    kb, qb, rb = oracle.round_to_bf16(k), oracle.round_to_bf16(q), oracle.round_to_bf16(R)
    P = oracle.round_to_bf16(np.eye(2, d, dtype=np.float32))
    T = np.arange(6, dtype=np.int32).reshape(2, 3)
    st = Store.of(kb, P, T)
    qsig, qamb = oracle.signatures(qb, rb)
    assert qamb[0, 0] and not qamb[1].any()
    assert oracle.hamming(qsig, oracle.signatures(kb, rb)[0])[0, 0] == 1
    _, amb = oracle.lookup_lsh(st, {"emb": qb, "prefix": P, "ids": T}, Params(0.9, 0.5, 2), rb, radius=0)
    assert amb.tolist() == [True, False]


def test_radius_zero_keeps_only_identical_signatures():
    st, qs = _small_case()
    R = wl.bf16_bits(wl.hyperplanes(64, 32))
    p = Params(0.9, 0.5, 8)
    qs = dict(qs, emb=st.key[:24].copy())                 # each query is an exact copy of entry j
    lsh, _ = oracle.lookup_lsh(st, qs, p, R, radius=0)
    qsig, _ = oracle.signatures(qs["emb"], R)
    esig, _ = oracle.signatures(st.key, R)
    same = oracle.hamming(qsig, esig) == 0
    for b in range(24):
        got = set(lsh.cand_id[b, :lsh.n_cand[b]].tolist())
        assert b in got and got <= set(np.nonzero(same[b])[0].tolist())


def test_suggested_radius_keeps_threshold_pairs():
    # at 4 standard deviations the binomial tail at the threshold angle is below 1e-4
    scipy_stats = pytest.importorskip("scipy.stats")
    for tau, b in [(0.9, 256), (0.85, 128), (0.88, 512)]:
        r = wl.lsh_radius(tau, b)
        assert scipy_stats.binom.sf(r, b, math.acos(tau) / math.pi) < 1e-4
