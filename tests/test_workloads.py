"""The seeded generator: determinism, chunk regeneration, and that its labels match the oracle's decisions."""
import numpy as np
import torch

import oracle
from paper_2608_01718_gb300 import workloads as wl


def _store_bits(w, device="cpu"):
    keys, pres, ids = [], [], []
    for ch in wl.iter_store(w, device):
        if w.key_dtype == "f32":
            keys.append(oracle.round_to_bf16(wl.f32_array(ch["key"])))
            pres.append(oracle.round_to_bf16(wl.f32_array(ch["prefix"])))
        else:
            keys.append(wl.bf16_bits(ch["key"]))
            pres.append(wl.bf16_bits(ch["prefix"]))
        ids.append(ch["ids"].numpy())
    return oracle.Store.of(np.concatenate(keys), np.concatenate(pres), np.concatenate(ids))


def test_deterministic_and_regenerable():
    w = wl.WORKLOADS["mid-1m"].scaled(n=wl.CHUNK_ROWS + 1000, d=64, batch=16)
    a = wl.store_chunk(w, 1)
    b = wl.store_chunk(w, 1)
    assert torch.equal(a["key"].view(torch.int16), b["key"].view(torch.int16))
    assert a["key"].shape == (1000, 64)
    rows = torch.tensor([3, wl.CHUNK_ROWS + 5, 7])
    got = wl.store_rows(w, rows)
    c0 = wl.store_chunk(w, 0)
    assert torch.equal(got["key"][0].view(torch.int16), c0["key"][3].view(torch.int16))
    assert torch.equal(got["ids"][1], a["ids"][5])
    q1, q2 = wl.batch(w, 0), wl.batch(w, 0)
    assert torch.equal(q1["emb"].view(torch.int16), q2["emb"].view(torch.int16))
    assert not torch.equal(wl.batch(w, 1)["emb"].view(torch.int16), q1["emb"].view(torch.int16))


def test_mix_counts_and_zipf_targets():
    w = wl.WORKLOADS["large-16m"].scaled(n=100_000)
    plan = wl.query_plan(w)
    near, rand, coll = wl.class_counts(w)
    assert (near, rand, coll) == (64, 38, 26)
    assert int((plan["class"] == wl.NEAR).sum()) == near
    assert torch.all((plan["target"] >= 0) == (plan["class"] != wl.RANDOM))
    assert int(plan["target"].max()) < 100_000


def test_labels_predict_oracle_decisions_on_tiny_cache():
    """Sanity rate, not parity: near-duplicate -> HIT on its target, collision -> REJECT, random -> MISS_KEY."""
    w = wl.WORKLOADS["tiny-4k"]
    st = _store_bits(w)
    q = wl.batch(w, 0)
    res = oracle.lookup(st, {"emb": wl.bf16_bits(q["emb"]), "prefix": wl.bf16_bits(q["prefix"]),
                             "ids": q["ids"].numpy()}, oracle.Params(w.tau_c, w.tau_a, w.top_c))
    cls, tgt = q["class"].numpy(), q["target"].numpy()
    near, rnd, coll = cls == wl.NEAR, cls == wl.RANDOM, cls == wl.COLLISION
    assert np.all(res.status[near] == oracle.HIT) and np.all(res.entry_id[near] == tgt[near])
    assert np.all(res.status[coll] == oracle.REJECT)
    assert np.all(res.status[rnd] == oracle.MISS_KEY)
    # every near-duplicate and collision has a full candidate list (the target's cluster clears tau_c)
    assert np.all(res.n_cand[near | coll] == w.top_c)
    assert np.min(res.margin) > 2e-3


def test_ensemble_workload_labels_predict_oracle_decisions():
    """Sanity rate on a small ensemble cache: with all three checks, near-duplicates hit and both kinds of
    collision are rejected; with the first check alone the prefix-mimicking collisions get through."""
    w = wl.WORKLOADS["ensemble-1m"].scaled(n=4096, clusters=64, batch=64)
    st = _store_bits(w)
    q = wl.batch(w, 0)
    oq = {"emb": wl.bf16_bits(q["emb"]), "prefix": wl.bf16_bits(q["prefix"]), "ids": q["ids"].numpy()}
    cls, tgt = q["class"].numpy(), q["target"].numpy()
    ens = oracle.lookup(st, oq, oracle.Params(w.tau_c, 0.0, w.top_c, prefix_dims=w.prefix_dims,
                                              tau_a_models=w.tau_a_models))
    near, mimic, coll = cls == wl.NEAR, cls == wl.MIMIC, cls == wl.COLLISION
    assert mimic.sum() > 0
    assert np.all(ens.status[near] == oracle.HIT) and np.all(ens.entry_id[near] == tgt[near])
    assert np.all(ens.status[mimic | coll] == oracle.REJECT)
    first = oracle.lookup(st, oq, oracle.Params(w.tau_c, 0.0, w.top_c, prefix_dims=w.prefix_dims,
                                                tau_a_models=(w.tau_a_models[0], -2.0, -2.0)))
    assert np.all(first.status[mimic] == oracle.HIT)
    assert np.all(ens.prefix_scores[near, 0] > 0.9) and ens.prefix_scores.shape == (w.batch, 3)
