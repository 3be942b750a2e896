"""Pins of the oracle's threshold calibration (App. A.2): the nearest-rank percentile against the textbook
definition, the cap rule against the paper's printed table, and the pair similarities against closed forms."""
import json
import os

import numpy as np
import pytest

import oracle

from test_oracle_pins import bits

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_nearest_rank_textbook_values():
    # The standard worked example of the nearest-rank method on {15, 20, 35, 40, 50}.
    v = [35, 50, 15, 40, 20]
    assert [oracle.nearest_rank(v, p) for p in (5, 30, 40, 50, 100)] == [15, 20, 20, 35, 50]
    rng = np.random.default_rng(0)
    hundred = rng.permutation(np.arange(1, 101))
    assert oracle.nearest_rank(hundred, 5) == 5 and oracle.nearest_rank(hundred, 10) == 10
    assert oracle.nearest_rank(hundred, 0) == 1 and oracle.nearest_rank(np.arange(1, 21), 10) == 2


def _sims_with_percentile(value, percentile, n=500, seed=0):
    """n similarities whose nearest-rank percentile is exactly `value`."""
    rng = np.random.default_rng(seed)
    rank = int(np.ceil(percentile / 100 * n))
    below = value - rng.uniform(0.01, 0.3, rank - 1)
    above = value + rng.uniform(0.001, 0.2, n - rank)
    return rng.permutation(np.concatenate([below, [value], above]))


def test_cap_rule_reproduces_the_papers_table():
    with open(os.path.join(GOLDEN, "calibration_appA2.json")) as f:
        table = json.load(f)
    for key in ("tau_c", "tau_a"):
        spec = table[key]
        for i, row in enumerate(spec["rows"]):
            sims = _sims_with_percentile(row["p"], spec["percentile"], seed=i)
            p = oracle.nearest_rank(sims, spec["percentile"])
            assert p == row["p"]
            assert min(spec["cap"], p) == pytest.approx(row["tau"], abs=1e-12)


def test_pair_similarities_closed_form_and_calibrate():
    e = np.eye(4)
    x = np.array([e[0], e[0], [0.5, 0.5, 0.5, 0.5], e[1]])
    y = np.array([e[0], [0.75, 0.5, 0.25, 0.0], [0.5, 0.5, 0.5, 0.5], e[2]])
    s = oracle.pair_similarities(bits(x), bits(y))
    assert list(s) == [1.0, 0.75, 1.0, 0.0]
    tau, p = oracle.calibrate(bits(x), bits(y), 50, 0.8)      # rank ceil(2) = 2 -> 0.75
    assert (p, tau) == (0.75, 0.75)
    tau, p = oracle.calibrate(bits(x), bits(y), 100, 0.8)     # the largest, capped
    assert (p, tau) == (1.0, 0.8)
