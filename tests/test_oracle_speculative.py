"""Pins of the draft-verification bookkeeping (section 3.3, "Speculative Decoding"): a draft token is accepted
if P_f(t) >= P_g(t), from the first token on, and the first rejection hands decoding to the target model."""
import numpy as np

import oracle
from oracle import HIT, MISS_KEY, REJECT


def test_acceptance_stops_at_the_first_rejection():
    pf = [[0.9, 0.8, 0.1, 0.9],      # third token rejected: 2 reused
          [0.2, 0.9, 0.9, 0.9],      # first token rejected: none reused
          [0.5, 0.5, 0.5, 0.5]]      # equal probabilities are accepted (>=): all 4 reused
    pg = [[0.5, 0.8, 0.2, 0.1],
          [0.3, 0.1, 0.1, 0.1],
          [0.5, 0.5, 0.5, 0.5]]
    assert list(oracle.accepted_prefix(pf, pg)) == [2, 0, 4]


def test_served_queries_verify_nothing():
    pf = np.full((3, 2), 0.9)
    pg = np.full((3, 2), 0.1)
    status = np.array([HIT, MISS_KEY, REJECT], np.uint8)
    assert list(oracle.accepted_prefix(pf, pg, status)) == [-1, 2, 2]


def test_accepted_length_is_the_first_failure_index():
    rng = np.random.default_rng(0)
    pf, pg = rng.random((500, 20)), rng.random((500, 20))
    got = oracle.accepted_prefix(pf, pg)
    fail = pf < pg
    want = np.where(fail.any(axis=1), fail.argmax(axis=1), 20)
    assert np.array_equal(got, want)
    # with independent uniform probabilities each token passes with probability 1/2: E[accepted] = 1 - 2^-20
    assert abs(got.mean() - (1 - 2.0 ** -20)) < 0.2
