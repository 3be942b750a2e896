"""Parity on seeded random configurations: each case draws the shapes and settings the fixed cases pin one at a time
(embedding width, window k, candidate list size, batch size, store size, thresholds, check mode, stage-1 kernel) and
compares the lookup through the C ABI with the fp64 oracle on the same bytes, under the usual rules (exact outside
the 2e-3 decision margin; an in-band HIT must still pass both checks)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

from parity import compare, fill, gpu_lookup, log_report, new_cache, oracle_queries, oracle_store, pair_scores_fn, params

pytestmark = pytest.mark.gpu

KERNELS = [L.LACACHE_STAGE1_AUTO, L.LACACHE_STAGE1_TENSOR, L.LACACHE_STAGE1_STREAM]


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


def _draw(seed):
    rng = np.random.default_rng(20261202 + seed)
    d = int(rng.choice([8, 24, 64, 136, 256, 384, 520, 768, 1024, 1536]))
    k = int(rng.integers(1, 65))
    top_c = int(rng.choice([1, 2, 3, 5, 8, 13, 16, 32]))
    batch = int(rng.choice([1, 2, 3, 4, 7, 16, 33, 100, 129, 200]))
    n = int(rng.choice([0, 1, 7, 300, 2049, 9000, 25000, 70000]))
    clusters = int(rng.choice([8, 64, 500]))
    tau_c = float(rng.choice([0.5, 0.8, 0.88, 0.9, 0.95]))
    tau_a = float(rng.choice([0.5, 0.7, 0.8, 0.9]))
    mode = int(rng.choice([oracle.CHECK_EMB, oracle.CHECK_TOKENS, oracle.CHECK_BOTH]))
    tmin = int(rng.integers(1, k + 1)) if mode != oracle.CHECK_EMB and rng.random() < 0.5 else None
    stage1 = KERNELS[int(rng.integers(0, len(KERNELS)))]
    w = wl.WORKLOADS["mid-1m"].scaled(n=n, d=d, k=k, top_c=top_c, batch=batch, clusters=clusters, tau_c=tau_c,
                                      tau_a=tau_a, vocab=int(rng.choice([3, 50, 128256])))
    return w, mode, tmin, stage1


@pytest.mark.parametrize("seed", range(40))
def test_random_configuration_matches_the_oracle(seed):
    w, mode, tmin, stage1 = _draw(seed)
    st = oracle_store(w) if w.n else None
    with new_cache(w, stage1, capacity=max(1, w.n), check_mode=mode, token_match_min=tmin or 0) as cache:
        if w.n:
            fill(cache, w)
        assert cache.size == w.n
        # an empty store's queries are drawn against a one-entry store that is never inserted
        q = wl.batch(w if w.n else w.scaled(n=1), 0, device="cuda")
        g = gpu_lookup(cache, q)
    p = params(w, mode, tmin)
    oq = oracle_queries(q)
    if st is None:
        assert np.all(g["status"] == oracle.MISS_KEY) and np.all(g["entry_id"] == -1)
        assert np.all(np.isneginf(g["key_score"])) and np.all(g["n_cand"] == 0)
        return
    res = oracle.lookup(st, oq, p)
    rep = compare(g, res, p, pair_scores=pair_scores_fn(st, oq))
    log_report(f"random seed={seed} n={w.n} d={w.d} k={w.k} c={w.top_c} B={w.batch} mode={mode} tmin={tmin} "
               f"stage1={stage1}", rep)
    assert rep.exact + rep.band == w.batch
