"""Entry-range sharding on one GPU: a store cut into G row ranges, one handle per range, each handle's lookup
written into its rank's slice of one gathered buffer (as the all-gather of paper_2608_01718_gb300.sharded leaves
it), then lacache_merge_shards. The merge must reproduce a single whole-store handle's lookup bit for bit, every
field including the candidate lists. A row's fp32 scores do not depend on which handle or tile holds it. The
merge must also match the oracle. The shard handles run one after another: no kernel waits on another."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01718_gb300 import build, sharded
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl
from parity import compare, log_report, new_cache, oracle_queries, oracle_store, params, fill

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


def fill_range(cache, w, a, b):
    """Insert store rows [a, b) of the workload."""
    dtype = L.LACACHE_F32 if w.key_dtype == "f32" else L.LACACHE_BF16
    off = 0
    for ch in wl.iter_store(w, "cuda"):
        n = ch["key"].shape[0]
        lo, hi = max(a, off), min(b, off + n)
        if lo < hi:
            cache.insert(ch["key"][lo - off:hi - off], ch["prefix"][lo - off:hi - off], ch["ids"][lo - off:hi - off],
                         dtype)
        off += n
    torch.cuda.synchronize()


CASES = {
    "tiny-2": (wl.WORKLOADS["tiny-4k"], (0, 2048, 4096), L.LACACHE_STAGE1_TENSOR, oracle.CHECK_EMB),
    "tiny-empty-stream": (wl.WORKLOADS["tiny-4k"], (0, 700, 700, 2901, 4096), L.LACACHE_STAGE1_STREAM, oracle.CHECK_EMB),
    "tiny-16": (wl.WORKLOADS["tiny-4k"], tuple(range(0, 4097, 256)), L.LACACHE_STAGE1_TENSOR, oracle.CHECK_EMB),
    "tiny-tokens": (wl.WORKLOADS["tiny-4k"].scaled(n=3000, k=4, vocab=3, batch=48), (0, 1100, 3000),
                    L.LACACHE_STAGE1_TENSOR, oracle.CHECK_TOKENS),
    "mid-4": (wl.WORKLOADS["mid-1m"].scaled(n=70_000), (0, 9000, 30_000, 51_234, 70_000), L.LACACHE_STAGE1_TENSOR,
              oracle.CHECK_EMB),
    "pairs-3": (wl.WORKLOADS["serve-2m"].scaled(n=12_050, batch=300, clusters=120), (0, 4000, 8000, 12_050),
                L.LACACHE_STAGE1_TENSOR, oracle.CHECK_EMB),
    "ensemble-2": (wl.WORKLOADS["ensemble-1m"].scaled(n=20_000, batch=48), (0, 7777, 20_000), L.LACACHE_STAGE1_TENSOR,
                   oracle.CHECK_EMB),
}


@pytest.mark.parametrize("case", list(CASES))
def test_merged_shards_equal_the_whole_store_lookup(case):
    w, cuts, stage1, mode = CASES[case]
    models = len(w.prefix_dims) if w.prefix_dims is not None else 1
    B, c = w.batch, w.top_c
    q = wl.batch(w, 0, device="cuda")
    with new_cache(w, stage1, check_mode=mode) as whole:
        fill(whole, w)
        ref = alloc = L.alloc_result(B, c, "cuda", candidates=True, models=models if models > 1 else 0)
        whole.lookup(q["emb"], q["prefix"], q["ids"], out=alloc)
        torch.cuda.synchronize()
        whole.sync()
    G = len(cuts) - 1
    gathered = torch.zeros((G, sharded.record_bytes(B, c, models)), dtype=torch.uint8, device="cuda")
    shards = []
    for g, (a, b) in enumerate(zip(cuts, cuts[1:])):
        with new_cache(w, stage1, check_mode=mode, capacity=max(1, b - a)) as part:
            fill_range(part, w, a, b)
            rec = sharded.views(gathered[g], B, c, models)
            out = {**L.alloc_result(B, c, "cuda", candidates=False), **rec}
            part.lookup(q["emb"], q["prefix"], q["ids"], out=out)
            torch.cuda.synchronize()
            part.sync()
        shards.append((rec, a))
    merged = L.alloc_result(B, c, "cuda", candidates=True, models=models if models > 1 else 0)
    L.lacache_merge_shards(shards, c, models, merged)
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in merged.items()}
    want = {k: v.cpu().numpy() for k, v in ref.items()}
    assert got.keys() == want.keys()
    for k in want:
        assert np.array_equal(got[k], want[k], equal_nan=True), k
    # and against the oracle, as every lookup is
    p = params(w, mode)
    res = oracle.lookup(oracle_store(w), oracle_queries(q), p)
    rep = compare(got, res, p)
    log_report(f"{case}: {G} shards merged, n={w.n} B={B}", rep)
    assert rep.exact + rep.band == B
    assert len({int(s) for s in got["status"]}) >= 2


def test_merge_rejects_bad_arguments():
    B, c = 4, 2
    rec = sharded.views(torch.zeros(sharded.record_bytes(B, c, 1), dtype=torch.uint8, device="cuda"), B, c, 1)
    out = L.alloc_result(B, c, "cuda")
    no_models = {k: v for k, v in rec.items() if k != "cand_prefix_scores"}
    for shards, models in [([], 1), ([(rec, 0)] * 17, 1), ([(rec, 10), (rec, 5)], 1), ([(no_models, 0)], 2),
                           ([(rec, -1)], 1), ([(rec, 0)], 9)]:
        with pytest.raises(L.LacacheError) as e:
            L.lacache_merge_shards(shards, c, models, out)
        assert e.value.status == L.LACACHE_ERR_INVALID_ARG


def test_merged_key_score_when_a_shard_hit_falls_past_the_cut():
    # query e0, top_c 2; shard A holds entries scoring 1 and 0.9375, shard B 0.984375 and 0.96875. Only entry 1
    # (0.9375) passes the lookahead check: shard A serves it, but globally it is third, past the cut. The merged
    # result is the whole store's: a REJECT of candidates [0, 2] whose key score is the best one, 1.
    d, B, c = 64, 1, 2
    eye = torch.eye(d, dtype=torch.float32)
    keys = torch.zeros((4, d))
    keys[:, 0] = torch.tensor([1.0, 0.9375, 0.984375, 0.96875])
    pres = torch.stack([eye[2], eye[1], eye[2], eye[2]])
    ids = torch.zeros((4, 1), dtype=torch.int32)
    q = {"emb": eye[:1].to(torch.bfloat16).cuda(), "prefix": eye[1:2].to(torch.bfloat16).cuda(),
         "ids": torch.zeros((1, 1), dtype=torch.int32, device="cuda")}
    gathered = torch.zeros((2, sharded.record_bytes(B, c, 1)), dtype=torch.uint8, device="cuda")
    shards, own = [], []
    for g, (a, b) in enumerate([(0, 2), (2, 4)]):
        with L.LaCache(d, 1, 2, 0.5, 0.5, c, max_batch=4) as part:
            part.insert(keys[a:b].to(torch.bfloat16).cuda(), pres[a:b].to(torch.bfloat16).cuda(), ids[a:b].cuda())
            rec = sharded.views(gathered[g], B, c, 1)
            out = {**L.alloc_result(B, c, "cuda", candidates=False), **rec}
            part.lookup(q["emb"], q["prefix"], q["ids"], out=out)
            torch.cuda.synchronize()
            own.append((int(out["status"][0]), float(out["key_score"][0])))
        shards.append((rec, a))
    assert own[0] == (L.LACACHE_HIT, 0.9375) and own[1] == (L.LACACHE_REJECT, 0.984375)
    merged = L.alloc_result(B, c, "cuda", candidates=True)
    L.lacache_merge_shards(shards, c, 1, merged)
    torch.cuda.synchronize()
    assert int(merged["status"][0]) == L.LACACHE_REJECT and float(merged["key_score"][0]) == 1.0
    assert merged["cand_id"][0].tolist() == [0, 2] and int(merged["entry_id"][0]) == -1
    assert float(merged["prefix_score"][0]) == 0.0


def test_merged_simhash_shards_equal_the_whole_store_lookup():
    # every shard signs its own rows with the same hyperplanes, so each admits exactly its part of the whole
    # store's admitted pairs: the merge equals the whole-store lookup through the index
    w = wl.WORKLOADS["mid-1m"].scaled(n=30_000, batch=16)
    cuts = (0, 11_111, 30_000)
    bits = 256
    radius = wl.lsh_radius(w.tau_c, bits)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    B, c = w.batch, w.top_c
    q = wl.batch(w, 0, device="cuda")
    with new_cache(w, L.LACACHE_STAGE1_LSH) as whole:
        fill(whole, w)
        L.lacache_enable_lsh(whole.h, bits, radius, R)
        ref = L.alloc_result(B, c, "cuda", candidates=True)
        whole.lookup(q["emb"], q["prefix"], q["ids"], out=ref)
        torch.cuda.synchronize()
        whole.sync()
    gathered = torch.zeros((len(cuts) - 1, sharded.record_bytes(B, c, 1)), dtype=torch.uint8, device="cuda")
    shards = []
    for g, (a, b) in enumerate(zip(cuts, cuts[1:])):
        with new_cache(w, L.LACACHE_STAGE1_LSH, capacity=b - a) as part:
            fill_range(part, w, a, b)
            L.lacache_enable_lsh(part.h, bits, radius, R)
            rec = sharded.views(gathered[g], B, c, 1)
            part.lookup(q["emb"], q["prefix"], q["ids"], out={**L.alloc_result(B, c, "cuda", candidates=False), **rec})
            torch.cuda.synchronize()
            part.sync()
        shards.append((rec, a))
    merged = L.alloc_result(B, c, "cuda", candidates=True)
    L.lacache_merge_shards(shards, c, 1, merged)
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in merged.items()}
    for k, v in ref.items():
        assert np.array_equal(got[k], v.cpu().numpy(), equal_nan=True), k
    p = params(w)
    res, amb = oracle.lookup_lsh(oracle_store(w), oracle_queries(q), p, wl.bf16_bits(R), radius)
    keep = np.nonzero(~amb)[0]
    rep = compare(got, oracle.Result(**{f: getattr(res, f)[keep] for f in res.__dataclass_fields__}), p, rows=keep)
    log_report(f"simhash: {len(cuts) - 1} shards merged, n={w.n} B={B}", rep)
    assert rep.exact + rep.band == len(keep) and len(keep) >= B - 1
