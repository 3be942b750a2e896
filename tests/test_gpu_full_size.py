"""Parity at the full sizes of the large workloads, in the launch configuration the benchmark uses.

large-16m (70 GB store) checks its whole batch of 128 queries against the streamed oracle, through the exact scan
and through the SimHash index, and batch-4m a stratified sample of 513 of its 8192 queries. serve-2m runs all 1000 steps. The oracle replays steps 0-2 from its
own state. Five seeded later steps are verified against the store rebuilt from the GPU's append log: every logged
row is first checked, bit for bit, against the non-HIT query row the GPU reported. Every step is also checked for
the properties that hold at any size: the append log, bit-exact appended rows, and both checks passing for every
HIT on a sampled step.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

from parity import (TOL, Report, StreamedOracle, compare, fill, log_report, new_cache, oracle_queries, oracle_store,
                    params, stratified_sample)

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


def _check_streamed(w, per_class, pairs_of_queries=False):
    """The full-size lookup of the whole batch (AUTO: the tensor-core scan), and with pairs_of_queries the same
    queries looked up two at a time (AUTO: the streaming scan at d = 1024), against the streamed oracle."""
    q = wl.batch(w, 0, device="cuda")
    sample = stratified_sample(q["class"], per_class)
    p = params(w)
    so = StreamedOracle(w, q, sample, p)
    small = None
    with new_cache(w, L.LACACHE_STAGE1_AUTO) as cache:
        so.fill(cache)
        assert cache.size == w.n
        out = cache.lookup(q["emb"], q["prefix"], q["ids"])
        torch.cuda.synchronize()
        cache.sync()
        # batches of more than one query tile run on CTA pairs
        assert cache.last_launch()[1] == (L.LACACHE_STAGE1_TENSOR_PAIR if w.batch > 128 else L.LACACHE_STAGE1_TENSOR)
        g = {k: v.cpu().numpy() for k, v in out.items()}
        if pairs_of_queries:
            parts = []
            for i in range(0, w.batch, 2):
                qq = {k: q[k][i:i + 2].contiguous() for k in ("emb", "prefix", "ids")}
                parts.append(cache.lookup(qq["emb"], qq["prefix"], qq["ids"]))
                assert cache.last_launch()[1] == L.LACACHE_STAGE1_STREAM
            torch.cuda.synchronize()
            cache.sync()
            small = {k: torch.cat([o[k] for o in parts]).cpu().numpy() for k in parts[0]}
    res = so.result()
    rep = compare(g, res, p, rows=sample, pair_scores=so.pair_scores)
    log_report(f"{w.name} full size, sampled", rep)
    if small is not None:
        rep2 = compare(small, res, p, rows=sample, pair_scores=so.pair_scores)
        log_report(f"{w.name} full size, two queries per lookup (streaming scan)", rep2)
        assert rep2.exact + rep2.band == len(sample) and rep2.band <= max(1, len(sample) // 50)
    assert rep.exact + rep.band == len(sample)
    assert rep.band <= max(1, len(sample) // 50)
    assert rep.hits > 0 and rep.rejects > 0 and rep.misses > 0
    # the generator's labels, as a sanity rate over the whole batch (not parity)
    cls, tgt = q["class"].numpy(), q["target"].numpy()
    near = cls == wl.NEAR
    assert np.mean(g["entry_id"][near] == tgt[near]) >= 0.99
    assert np.mean(g["status"][cls == wl.COLLISION] == L.LACACHE_REJECT) >= 0.99
    return rep


def test_large_cache_near_hbm_capacity():
    """16,777,216 entries x 1024 dims (34 GB of keys), B = 128, Zipf(1.1) targets: every query of the batch."""
    rep = _check_streamed(wl.WORKLOADS["large-16m"], per_class=128, pairs_of_queries=True)
    assert rep.queries == 128


def test_large_cache_through_the_simhash_index():
    """16,777,216 entries x 1024 looked up through a 256-bit SimHash index (B = 128: the tensor-core Hamming scan
    over the expanded index), every query of the batch against the streamed oracle. Queries whose outcome an
    ambiguous signature bit could change are set aside (at most 1 in 50)."""
    w = wl.WORKLOADS["large-16m"]
    bits = 256
    radius = wl.lsh_radius(w.tau_c, bits)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    q = wl.batch(w, 0, device="cuda")
    sample = np.arange(w.batch)
    p = params(w)
    so = StreamedOracle(w, q, sample, p, lsh=(wl.bf16_bits(R), radius))
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        so.fill(cache)
        L.lacache_enable_lsh(cache.h, bits, radius, R)
        out = cache.lookup(q["emb"], q["prefix"], q["ids"])
        torch.cuda.synchronize()
        cache.sync()
        assert cache.last_launch()[1] == L.LACACHE_STAGE1_LSH_TENSOR
        g = {k: v.cpu().numpy() for k, v in out.items()}
    res = so.result()
    keep = np.nonzero(~so.ambiguous)[0]
    sub = oracle.Result(**{f: getattr(res, f)[keep] for f in res.__dataclass_fields__})
    rep = compare(g, sub, p, rows=sample[keep], pair_scores=lambda b, j: so.pair_scores(int(keep[b]), j))
    log_report(f"{w.name} full size through the SimHash index ({w.batch - len(keep)} queries with ambiguous bits)",
               rep)
    assert len(keep) >= w.batch - max(2, w.batch // 50)
    assert rep.exact + rep.band == len(keep) and rep.band <= max(1, len(keep) // 50)
    assert rep.hits > 0 and rep.rejects > 0 and rep.misses > 0


def test_large_batch_tensor_core_regime():
    """4,194,304 entries x 768, B = 8192 (64 query tiles), top_c = 16: 171 queries of each class."""
    rep = _check_streamed(wl.WORKLOADS["batch-4m"], per_class=171)
    assert rep.queries >= 512


def test_serve_loop_thousand_steps():
    """2,097,152 initial entries, 1000 batches of 256, every miss appended (about 2.24M entries at the end)."""
    w = wl.WORKLOADS["serve-2m"]
    capacity = w.n + w.steps * w.batch
    p = params(w)
    replay = 3
    later = set(np.random.default_rng(w.seed).choice(np.arange(replay, w.steps), size=5, replace=False).tolist())
    st = oracle_store(w)
    # the oracle's own store: its appends on the replayed steps, then the rows of the GPU's append log
    loop = oracle.ServeLoop(capacity, w.d, w.k, p)
    loop.insert(st.key, st.prefix, st.ids)
    del st
    origin = {}          # appended entry id -> (step, query index) of the query it holds
    hits_checked = 0
    replayed = Report()
    rebuilt = Report()
    with new_cache(w, L.LACACHE_STAGE1_TENSOR, capacity=capacity) as cache:
        fill(cache, w)
        for step in range(w.steps):
            q = wl.batch(w, step, device="cuda")
            n_before = cache.size
            out = cache.lookup(q["emb"], q["prefix"], q["ids"])
            first, m = cache.append_misses(q["emb"], q["prefix"], q["ids"], out["status"])
            status = out["status"].cpu().numpy()
            miss = np.nonzero(status != L.LACACHE_HIT)[0]
            assert first == n_before and m == len(miss) and cache.size == n_before + m
            # the appended rows are the non-HIT queries of this step, in query order, bit for bit
            key = torch.empty((m, w.d), dtype=torch.bfloat16, device="cuda")
            pre = torch.empty_like(key)
            ids = torch.empty((m, w.k), dtype=torch.int32, device="cuda")
            L.lacache_read_rows(cache.h, first, m, key=key, prefix=pre, ids=ids)
            sel = torch.as_tensor(miss, device="cuda")
            assert torch.equal(key.view(torch.int16), q["emb"][sel].view(torch.int16))
            assert torch.equal(pre.view(torch.int16), q["prefix"][sel].view(torch.int16))
            assert torch.equal(ids, q["ids"][sel])
            origin.update({first + i: (step, int(qi)) for i, qi in enumerate(miss)})
            oq = oracle_queries(q)
            if step < replay:
                g = {k: v.cpu().numpy() for k, v in out.items()}
                res, ofirst, om = loop.step(oq)
                rep = compare(g, res, p)
                replayed.add(rep)
                assert rep.band == 0 and (ofirst, om) == (first, m)
            else:
                assert loop.n == n_before
                if step in later:
                    # this step's decisions, verified against the store as the append log left it
                    g = {k: v.cpu().numpy() for k, v in out.items()}
                    rep = compare(g, oracle.lookup(loop.store, oq, p), p)
                    rebuilt.add(rep)
                    assert rep.band <= max(1, w.batch // 50)
                # the logged rows (checked above against the reported non-HIT queries) join the oracle's store
                loop.insert(oq["emb"][miss], oq["prefix"][miss], oq["ids"][miss])
            if step % 97 == 0:
                hits_checked += _check_hits(w, p, q, out, origin)
        assert cache.size > w.n + 100 * w.steps
        assert hits_checked > 100
    log_report(f"{w.name} oracle-replayed steps 0-{replay - 1}", replayed)
    log_report(f"{w.name} steps {sorted(later)} against the store rebuilt from the append log", rebuilt)
    assert rebuilt.queries == 5 * w.batch and rebuilt.hits > 0 and rebuilt.rejects > 0 and rebuilt.misses > 0
    print(f"PARITY {w.name}: {w.steps} steps, final size {w.n + len(origin)}, HITs checked {hits_checked}",
          flush=True)


def _check_hits(w, p, q, out, origin):
    """Every HIT passes both checks against its entry's row, regenerated from the generator."""
    status = out["status"].cpu().numpy()
    hit = np.nonzero(status == L.LACACHE_HIT)[0]
    ent = out["entry_id"].cpu().numpy()[hit]
    oq = oracle_queries(q, torch.as_tensor(hit))
    initial = ent < w.n
    rows_k = np.zeros((len(hit), w.d), np.uint16)
    rows_p = np.zeros((len(hit), w.d), np.uint16)
    if initial.any():
        r = wl.store_rows(w, torch.as_tensor(ent[initial]), "cuda")
        rows_k[initial], rows_p[initial] = wl.bf16_bits(r["key"]), wl.bf16_bits(r["prefix"])
    for i in np.nonzero(~initial)[0]:
        step, qi = origin[int(ent[i])]
        src = wl.batch(w, step, device="cuda")
        rows_k[i], rows_p[i] = wl.bf16_bits(src["emb"][qi:qi + 1])[0], wl.bf16_bits(src["prefix"][qi:qi + 1])[0]
    for i in range(len(hit)):
        kc = oracle.KeyCheck(oq["emb"][i:i + 1], -np.inf)
        kc.add_rows(rows_k[i:i + 1], 0)
        r, _ = oracle.lookahead(oq["prefix"][i], oq["ids"][i], rows_p[i:i + 1], oq["ids"][i:i + 1])
        assert kc.best[0] >= p.tau_c - TOL and r[0] >= p.tau_a - TOL
    return len(hit)
