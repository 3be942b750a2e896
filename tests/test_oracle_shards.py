"""Entry-range sharding on the CPU: the oracle's merge of per-shard lookups is pinned to the whole-store lookup
(a separate computation over the same rows), and the rank exchange of paper_2608_01718_gb300.sharded runs over
two gloo ranks."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2608_01718_gb300 import sharded
from paper_2608_01718_gb300 import workloads as wl

EXACT = ("entry_id", "status", "n_cand", "cand_id", "cand_matches", "token_matches", "cand_pass")
CLOSE = ("key_score", "prefix_score", "cand_score", "cand_prefix_score", "prefix_scores", "cand_prefix_scores")


def _store(w):
    keys, pres, ids = [], [], []
    for ch in wl.iter_store(w, "cpu"):
        if w.key_dtype == "f32":
            keys.append(oracle.round_to_bf16(wl.f32_array(ch["key"])))
            pres.append(oracle.round_to_bf16(wl.f32_array(ch["prefix"])))
        else:
            keys.append(wl.bf16_bits(ch["key"]))
            pres.append(wl.bf16_bits(ch["prefix"]))
        ids.append(ch["ids"].numpy())
    return oracle.Store.of(np.concatenate(keys), np.concatenate(pres), np.concatenate(ids))


def _queries(w):
    q = wl.batch(w, 0)
    return {"emb": wl.bf16_bits(q["emb"]), "prefix": wl.bf16_bits(q["prefix"]), "ids": q["ids"].numpy()}


def _params(w, mode=oracle.CHECK_EMB):
    if w.prefix_dims is not None:
        return oracle.Params(w.tau_c, 0.0, w.top_c, check_mode=mode, prefix_dims=w.prefix_dims,
                             tau_a_models=w.tau_a_models)
    return oracle.Params(w.tau_c, w.tau_a, w.top_c, check_mode=mode)


def _sub(st, a, b):
    return oracle.Store.of(st.key[a:b], st.prefix[a:b], st.ids[a:b])


def _assert_same(merged, whole, fields_exact=EXACT):
    for f in fields_exact:
        np.testing.assert_array_equal(getattr(merged, f), getattr(whole, f), err_msg=f)
    for f in CLOSE:
        np.testing.assert_allclose(getattr(merged, f), getattr(whole, f), rtol=0, atol=1e-12, equal_nan=True,
                                   err_msg=f)


@pytest.mark.parametrize("cuts", [(0, 4096), (0, 2048, 4096), (0, 700, 700, 2901, 4096),
                                  (0, 819, 1638, 2457, 3276, 4096)], ids=["1", "2", "3+empty", "5"])
@pytest.mark.parametrize("mode", [oracle.CHECK_EMB, oracle.CHECK_TOKENS, oracle.CHECK_BOTH])
def test_merge_of_shards_equals_whole_store_lookup(cuts, mode):
    w = wl.WORKLOADS["tiny-4k"]
    st, oq, p = _store(w), _queries(w), _params(w, mode)
    whole = oracle.lookup(st, oq, p)
    parts = [oracle.lookup(_sub(st, a, b), oq, p) for a, b in zip(cuts, cuts[1:])]
    merged = oracle.merge_shards(parts, list(cuts[:-1]), p)
    _assert_same(merged, whole)
    np.testing.assert_array_equal(merged.n_above, whole.n_above)
    if len(cuts) > 2:
        # the case is not degenerate: some candidate lists draw on several shards, and some shards cut their own
        # lists at top_c
        shard_of = np.searchsorted(np.asarray(cuts[1:]), merged.cand_id, side="right")
        spans = [len(set(shard_of[b, :merged.n_cand[b]])) for b in range(len(merged.status))]
        assert max(spans) >= 2
        assert any(np.any(r.n_above > p.top_c) for r in parts)
    assert {oracle.HIT, oracle.REJECT, oracle.MISS_KEY} <= set(np.unique(merged.status))


def test_merge_of_ensemble_shards():
    w = wl.WORKLOADS["ensemble-1m"].scaled(n=4096, clusters=64, batch=64)
    st, oq, p = _store(w), _queries(w), _params(w)
    whole = oracle.lookup(st, oq, p)
    cuts = (0, 1500, 4096)
    parts = [oracle.lookup(_sub(st, a, b), oq, p) for a, b in zip(cuts, cuts[1:])]
    _assert_same(oracle.merge_shards(parts, list(cuts[:-1]), p), whole)


@pytest.mark.parametrize("dup_at", [3000, 5], ids=["later shard", "earlier shard"])
def test_equal_scores_across_shards_order_by_global_id(dup_at):
    # the served target of a near-duplicate query is copied, key, prefix and ids, to another row in another
    # shard: the two entries tie exactly, and the lower global id comes first
    w = wl.WORKLOADS["tiny-4k"]
    st, oq, p = _store(w), _queries(w), _params(w)
    whole0 = oracle.lookup(st, oq, p)
    # a HIT whose target lies in the other shard than dup_at
    b = next(b for b in np.nonzero(whole0.status == oracle.HIT)[0] if (whole0.entry_id[b] < 2048) != (dup_at < 2048))
    j = int(whole0.entry_id[b])
    for arr in (st.key, st.prefix, st.ids):
        arr[dup_at] = arr[j]
    whole = oracle.lookup(st, oq, p)
    i = list(whole.cand_id[b]).index(min(j, dup_at))
    assert whole.cand_id[b, i + 1] == max(j, dup_at) and whole.cand_score[b, i] == whole.cand_score[b, i + 1]
    parts = [oracle.lookup(_sub(st, 0, 2048), oq, p), oracle.lookup(_sub(st, 2048, 4096), oq, p)]
    merged = oracle.merge_shards(parts, [0, 2048], p)
    _assert_same(merged, whole)
    assert merged.entry_id[b] == min(j, dup_at)


def test_merged_key_score_is_the_best_over_shards_when_a_shard_hit_falls_past_the_cut():
    # query e0, top_c 2, entries scoring 1, 0.9375 (shard A, ids 0-1) and 0.984375, 0.96875 (shard B, ids 2-3).
    # Only entry 1 passes the lookahead check. Shard A serves it (a HIT reporting key score 0.9375), but globally
    # it is third, past the cut: the whole-store result is a REJECT whose key score is the best one, 1.
    E4 = np.eye(4)
    keys = [[1.0, 0, 0, 0], [0.9375, 0, 0, 0], [0.984375, 0, 0, 0], [0.96875, 0, 0, 0]]
    st = oracle.Store.of(oracle.round_to_bf16(np.array(keys, np.float32)),
                         oracle.round_to_bf16(np.array([E4[2], E4[1], E4[2], E4[2]], np.float32)),
                         np.zeros((4, 1), np.int32))
    oq = {"emb": oracle.round_to_bf16(E4[:1].astype(np.float32)),
          "prefix": oracle.round_to_bf16(E4[1:2].astype(np.float32)), "ids": np.zeros((1, 1), np.int32)}
    p = oracle.Params(0.5, 0.5, 2)
    whole = oracle.lookup(st, oq, p)
    parts = [oracle.lookup(_sub(st, 0, 2), oq, p), oracle.lookup(_sub(st, 2, 4), oq, p)]
    assert parts[0].status[0] == oracle.HIT and parts[0].key_score[0] == 0.9375
    assert whole.status[0] == oracle.REJECT and whole.key_score[0] == 1.0 and list(whole.cand_id[0]) == [0, 2]
    merged = oracle.merge_shards(parts, [0, 2], p)
    _assert_same(merged, whole)


def test_merge_rejects_mismatched_bases():
    w = wl.WORKLOADS["tiny-4k"]
    st, oq, p = _store(w), _queries(w), _params(w)
    with pytest.raises(ValueError):
        oracle.merge_shards([oracle.lookup(st, oq, p)], [0, 10], p)


def test_record_layout_is_aligned_and_views_cover_it():
    fields, size = sharded.layout(32, 8, 3)
    assert size % 16 == 0 and all(off % 16 == 0 for _, _, _, off in fields)
    buf = torch.zeros(size, dtype=torch.uint8)
    v = sharded.views(buf, 32, 8, 3)
    assert v["cand_prefix_scores"].shape == (32, 8, 3) and v["cand_pass"].dtype == torch.uint8
    v["n_cand"].fill_(-1)   # views alias the buffer and do not overlap the other fields
    assert int((buf != 0).sum()) == 32 * 4
    # four [32 x 8] 4-byte arrays, [32 x 8 x 1] scores, two [32] arrays, [32 x 8] pass bytes
    assert sharded.record_bytes(32, 8, 1) == 4 * 1024 + 1024 + 2 * 128 + 256
    with pytest.raises(ValueError):
        sharded.views(torch.zeros(size + 16, dtype=torch.uint8), 32, 8, 3)


# ---- two gloo ranks, each holding half of the store -------------------------------------------------------------

def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _to_views(res, rec):
    rec["cand_id"].copy_(torch.from_numpy(res.cand_id))
    rec["cand_score"].copy_(torch.from_numpy(res.cand_score))
    rec["cand_prefix_score"].copy_(torch.from_numpy(res.cand_prefix_score))
    rec["cand_matches"].copy_(torch.from_numpy(res.cand_matches))
    rec["cand_prefix_scores"].copy_(torch.from_numpy(res.cand_prefix_scores))
    rec["key_score"].copy_(torch.from_numpy(res.key_score))
    rec["n_cand"].copy_(torch.from_numpy(res.n_cand))
    rec["cand_pass"].copy_(torch.from_numpy(res.cand_pass.astype(np.uint8)))


def _of_views(rec):
    B, c = rec["cand_id"].shape
    nan = np.full(B, np.nan)
    return oracle.Result(
        entry_id=np.full(B, -1, np.int32), status=np.zeros(B, np.uint8), key_score=rec["key_score"].numpy(),
        prefix_score=nan, token_matches=np.full(B, -1, np.int32), n_cand=rec["n_cand"].numpy(),
        n_above=rec["n_cand"].numpy().astype(np.int64), cand_id=rec["cand_id"].numpy(),
        cand_score=rec["cand_score"].numpy(), cand_prefix_score=rec["cand_prefix_score"].numpy(),
        cand_matches=rec["cand_matches"].numpy(),
        prefix_scores=np.full((B, rec["cand_prefix_scores"].shape[2]), np.nan),
        cand_pass=rec["cand_pass"].numpy().astype(bool), cand_prefix_scores=rec["cand_prefix_scores"].numpy(),
        margin=nan, list_margin=nan, literal_margin=nan, next_id=np.full(B, -1, np.int32), next_score=nan)


def _rank(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = wl.WORKLOADS["tiny-4k"]
        st, oq, p = _store(w), _queries(w), _params(w)
        a, b = w.n * rank // world, w.n * (rank + 1) // world
        mine = _sub(st, a, b)
        out = {}
        lk = sharded.ShardedLookup(
            w.batch, w.top_c, 1, a, "cpu",
            local_lookup=lambda queries, rec: _to_views(oracle.lookup(mine, queries, p), rec),
            merge=lambda shards, o: o.update(res=oracle.merge_shards([_of_views(v) for v, _ in shards],
                                                                     [base for _, base in shards], p)),
            float_dtype=torch.float64)
        lk(oq, out)
        whole = oracle.lookup(st, oq, p)
        _assert_same(out["res"], whole)
        results[rank] = (lk.bases, int((out["res"].status == oracle.HIT).sum()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_merge_to_the_whole_store_lookup():
    world = 2
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, world, port, results)) for r in range(world)]
        for pr in procs:
            pr.start()
        for pr in procs:
            pr.join(300)
            assert pr.exitcode == 0
        res = dict(results)
    assert res[0] == res[1] and res[0][0] == [0, 2048] and res[0][1] > 0


# ---- failure detection on the host: a rank that dies between lookups ---------------------------------------------

def _rank_that_may_die(rank, world, port, results):
    import datetime
    import time
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=10))
    w = wl.WORKLOADS["tiny-4k"]
    st, oq, p = _store(w), _queries(w), _params(w)
    a, b = w.n * rank // world, w.n * (rank + 1) // world
    mine = _sub(st, a, b)
    lk = sharded.ShardedLookup(
        w.batch, w.top_c, 1, a, "cpu",
        local_lookup=lambda queries, rec: _to_views(oracle.lookup(mine, queries, p), rec),
        merge=lambda shards, o: o.update(res=oracle.merge_shards([_of_views(v) for v, _ in shards],
                                                                 [base for _, base in shards], p)),
        float_dtype=torch.float64)
    out = {}
    lk(oq, out)                     # one lookup completes on both ranks
    if rank == 1:
        os._exit(3)                 # then this rank dies, with nothing of the next exchange started
    t0 = time.monotonic()
    try:
        lk(oq, out)
        results[rank] = ("completed", 0.0)
    except Exception as e:          # the exchange reports the lost peer instead of waiting forever
        results[rank] = (type(e).__name__, time.monotonic() - t0)


def test_a_dead_rank_fails_the_next_exchange_instead_of_hanging():
    world = 2
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank_that_may_die, args=(r, world, port, results)) for r in range(world)]
        for pr in procs:
            pr.start()
        for pr in procs:
            pr.join(120)
        codes = [pr.exitcode for pr in procs]
        res = dict(results)
    assert codes[1] == 3
    assert 0 in res and res[0][0] != "completed", res
    assert res[0][1] < 60.0, res    # bounded by the process group's timeout, not an indefinite wait
