"""Parity of the ensemble of lookahead checks (section 3.4: a hit needs every model's prefix similarity to clear
its threshold) on seeded random configurations: each case draws the number of models (2-8), each model's prefix
dimension and threshold, the noise on near-duplicates' prefixes, a mix with prefix-mimicking collisions, the store
size, d, the batch, top_c and the stage-1 kernel, and compares the lookup through the C ABI with the oracle under
the usual rules (exact outside the 2e-3 decision margin; an in-band HIT must still pass every check)."""
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
    rng = np.random.default_rng(20261204 + seed)
    m = int(rng.integers(2, 9))
    dims = tuple(int(rng.choice([8, 64, 384, 768, 1024])) for _ in range(m))
    taus = tuple(float(rng.choice([0.5, 0.7, 0.9])) for _ in range(m))
    w = wl.WORKLOADS["ensemble-1m"].scaled(
        n=int(rng.choice([300, 7000, 40_000])), d=int(rng.choice([256, 768])), batch=int(rng.choice([1, 8, 48, 200])),
        top_c=int(rng.choice([1, 8, 16])), clusters=int(rng.choice([8, 64, 500])), prefix_dims=dims,
        tau_a_models=taus, near_prefix_sigma=float(rng.choice([0.0, 0.3, 0.6])))
    return w, KERNELS[int(rng.integers(0, len(KERNELS)))]


@pytest.mark.parametrize("seed", range(16))
def test_random_ensemble_configuration_matches_the_oracle(seed):
    w, stage1 = _draw(seed)
    st = oracle_store(w)
    with new_cache(w, stage1) as cache:
        fill(cache, w)
        q = wl.batch(w, 0, device="cuda")
        g = gpu_lookup(cache, q)
    assert g["prefix_scores"].shape == (w.batch, len(w.prefix_dims))
    p = params(w)
    oq = oracle_queries(q)
    rep = compare(g, oracle.lookup(st, oq, p), p, pair_scores=pair_scores_fn(st, oq))
    log_report(f"random ensemble seed={seed} n={w.n} d={w.d} B={w.batch} c={w.top_c} dims={w.prefix_dims} "
               f"tau_a={w.tau_a_models} sigma={w.near_prefix_sigma} stage1={stage1}", rep)
    assert rep.exact + rep.band == w.batch


@pytest.mark.parametrize("seed", range(6))
def test_random_ensemble_through_the_simhash_index(seed):
    # the same ensembles, stage 1 through a SimHash index (the radius the threshold gives): stage 2's m checks
    # are independent of how the candidates were found
    w, _ = _draw(100 + seed)
    bits = (128, 256, 512)[seed % 3]
    radius = wl.lsh_radius(w.tau_c, bits)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    st = oracle_store(w)
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        L.lacache_enable_lsh(cache.h, bits, radius, R)
        q = wl.batch(w, 0, device="cuda")
        g = gpu_lookup(cache, q)
    p = params(w)
    res, amb = oracle.lookup_lsh(st, oracle_queries(q), p, wl.bf16_bits(R), radius)
    keep = np.nonzero(~amb)[0]
    sub = oracle.Result(**{f: getattr(res, f)[keep] for f in res.__dataclass_fields__})
    rep = compare(g, sub, p, rows=keep)
    log_report(f"random ensemble simhash seed={seed} n={w.n} B={w.batch} dims={w.prefix_dims} bits={bits}", rep)
    assert len(keep) >= w.batch - min(2, max(1, w.batch // 50))
    assert rep.exact + rep.band == len(keep)


def test_ensemble_host_lookups_and_appends():
    # an ensemble's prefix rows are pd = sum of the models' dims wide: host lookups stage them, appends copy them
    w = wl.WORKLOADS["ensemble-1m"].scaled(n=9000, batch=40, prefix_dims=(1024, 8, 384))
    assert w.pd == 1416
    with new_cache(w, L.LACACHE_STAGE1_TENSOR, capacity=w.n + 2 * w.batch) as cache:
        fill(cache, w)
        qs = [wl.batch(w, i, device="cuda") for i in range(2)]
        want = [gpu_lookup(cache, q) for q in qs]
        hq = [{k: q[k].cpu().pin_memory() for k in ("emb", "prefix", "ids")} for q in qs]
        outs = [L.alloc_result(w.batch, w.top_c, "cpu", pinned=True, models=3) for _ in qs]
        stream = torch.cuda.current_stream()
        for q, o in zip(hq, outs):
            L.lacache_lookup_host_async(cache.h, q["emb"], q["prefix"], q["ids"], o, stream)
        stream.synchronize()
        cache.sync()
        for o, g in zip(outs, want):
            for k, v in o.items():
                assert np.array_equal(v.numpy(), g[k], equal_nan=True), k
        q = qs[0]
        status = torch.as_tensor(want[0]["status"], device="cuda")
        first, m = cache.append_misses(q["emb"], q["prefix"], q["ids"], status)
        miss = torch.nonzero(status != L.LACACHE_HIT).flatten()
        assert m == len(miss) and m > 0
        key = torch.empty((m, w.d), dtype=torch.bfloat16, device="cuda")
        pre = torch.empty((m, w.pd), dtype=torch.bfloat16, device="cuda")
        ids = torch.empty((m, w.k), dtype=torch.int32, device="cuda")
        L.lacache_read_rows(cache.h, first, m, key=key, prefix=pre, ids=ids)
        torch.cuda.synchronize()
        assert torch.equal(key.view(torch.int16), q["emb"][miss].view(torch.int16))
        assert torch.equal(pre.view(torch.int16), q["prefix"][miss].view(torch.int16))
        assert torch.equal(ids, q["ids"][miss])
