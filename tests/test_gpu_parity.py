"""GPU parity: the CUDA lookup (through the C ABI) against the fp64 oracle on the same seeded bytes.

Both stage-1 kernels are covered (the tcgen05 tensor-core scan and the streaming CUDA-core scan). Cases span several key
tiles with a ragged tail, ragged query tiles and ragged k-steps, the empty cache, exact duplicates, inclusive
thresholds, top_c = 1 and 32, every check mode, host-buffer lookups and the serve loop with appends.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

from parity import (Report, compare, fill, gpu_lookup, log_report, new_cache, oracle_queries, oracle_store,
                    pair_scores_fn, params)

pytestmark = pytest.mark.gpu

PATHS = [pytest.param(L.LACACHE_STAGE1_TENSOR, id="tensor"), pytest.param(L.LACACHE_STAGE1_STREAM, id="stream")]


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


def expected_kernel(stage1, batch):
    """The tensor path runs batches of more than one query tile on CTA pairs."""
    return L.LACACHE_STAGE1_TENSOR_PAIR if stage1 == L.LACACHE_STAGE1_TENSOR and batch > 128 else stage1


def run_parity(w, stage1, check_mode=oracle.CHECK_EMB, token_match_min=None, steps=(0,)):
    st = oracle_store(w)
    rep = Report()
    with new_cache(w, stage1, check_mode=check_mode, token_match_min=token_match_min or 0) as cache:
        fill(cache, w)
        assert cache.size == w.n
        for step in steps:
            q = wl.batch(w, step, device="cuda")
            g = gpu_lookup(cache, q)
            splits, kernel = cache.last_launch()
            assert kernel == expected_kernel(stage1, w.batch) and splits >= 1
            oq = oracle_queries(q)
            p = params(w, check_mode, token_match_min)
            res = oracle.lookup(st, oq, p)
            rep.add(compare(g, res, p, pair_scores=pair_scores_fn(st, oq)))
    log_report(f"{w.name} n={w.n} B={w.batch} stage1={stage1} mode={check_mode}", rep)
    return rep


@pytest.mark.parametrize("stage1", PATHS)
def test_tiny_reference_cache(stage1):
    w = wl.WORKLOADS["tiny-4k"]
    rep = run_parity(w, stage1, steps=(0, 1))
    assert rep.band == 0 and rep.exact == 2 * w.batch
    assert rep.hits > 0 and rep.rejects > 0 and rep.misses > 0


@pytest.mark.parametrize("stage1", PATHS)
def test_mid_cache_scaled_ragged_tail(stage1):
    w = wl.WORKLOADS["mid-1m"].scaled(n=70_000)          # 273 full key tiles and a ragged one
    rep = run_parity(w, stage1)
    assert rep.exact + rep.band == w.batch and rep.band <= 1


@pytest.mark.parametrize("stage1", PATHS)
def test_ragged_batch_dimension_and_k(stage1):
    # B = 130: two query tiles, the second ragged; d = 200: the last k-step is ragged; k = 3; c = 5
    w = wl.WORKLOADS["mid-1m"].scaled(n=5_000, d=200, k=3, batch=130, top_c=5, clusters=50, vocab=7)
    rep = run_parity(w, stage1)
    assert rep.exact + rep.band == w.batch and rep.band <= 2


@pytest.mark.parametrize("stage1", PATHS)
@pytest.mark.parametrize("d,k,batch", [(8, 1, 1), (8192, 256, 40)], ids=["smallest", "largest"])
def test_dimension_and_window_extremes(stage1, d, k, batch):
    # the smallest dimension, window and batch a handle accepts, and the largest dimension and window: one k-step of
    # 8 elements against 128 k-steps, and 1 token id against 256 per candidate row
    w = wl.WORKLOADS["mid-1m"].scaled(n=3_000, d=d, k=k, batch=batch, clusters=30, vocab=5)
    rep = run_parity(w, stage1, steps=(0, 1))
    assert rep.exact + rep.band == 2 * w.batch


@pytest.mark.parametrize("d", [384, 768, 1024])
@pytest.mark.parametrize("batch", [1, 2, 3, 5, 8, 9, 17])
def test_stream_query_groups_and_load_phases(d, batch):
    """The streaming scan's shapes: query groups of 1, 2, 4 and 8 (the batch rounded up; several groups past 8),
    one or two load phases per row, lanes without a chunk (d = 384), and a store that is not a whole number of
    warp tiles or splits."""
    w = wl.WORKLOADS["mid-1m"].scaled(n=20_011, d=d, batch=batch)
    rep = run_parity(w, L.LACACHE_STAGE1_STREAM)
    assert rep.exact + rep.band == w.batch and rep.band <= 1


def test_auto_takes_the_stream_scan_only_for_small_batches_on_stores_l2_holds():
    """LACACHE_STAGE1_AUTO: the streaming scan while n d B <= 2^25, and for 1 or 2 queries at d = 1024, the
    tensor-core scan otherwise (and the oracle agrees with its results)."""
    tiny = wl.WORKLOADS["tiny-4k"].scaled(batch=22)                # 4,096 x 384: n d = 1,572,864
    small = wl.WORKLOADS["mid-1m"].scaled(n=10_000, batch=8)      # 15 MB of keys, n d = 7,680,000
    mid = wl.WORKLOADS["mid-1m"].scaled(n=20_000, batch=3)        # 30.7 MB of keys, n d = 15,360,000
    large = wl.WORKLOADS["mid-1m"].scaled(n=30_000, batch=8)      # 46 MB of keys, n d = 23,040,000
    over = wl.WORKLOADS["mid-1m"].scaled(n=44_000, batch=2)       # 68 MB of keys, n d = 33,792,000 > 2^25
    wide = wl.WORKLOADS["large-16m"].scaled(n=30_000, batch=8)    # d = 1024, 61 MB of keys
    for w, want in ((tiny, {16: L.LACACHE_STAGE1_STREAM, 21: L.LACACHE_STAGE1_STREAM, 22: L.LACACHE_STAGE1_TENSOR}),
                    (small, {1: L.LACACHE_STAGE1_STREAM, 4: L.LACACHE_STAGE1_STREAM, 5: L.LACACHE_STAGE1_TENSOR}),
                    (mid, {2: L.LACACHE_STAGE1_STREAM, 3: L.LACACHE_STAGE1_TENSOR}),
                    (large, {1: L.LACACHE_STAGE1_STREAM, 2: L.LACACHE_STAGE1_TENSOR, 4: L.LACACHE_STAGE1_TENSOR}),
                    (over, {1: L.LACACHE_STAGE1_TENSOR}),
                    (wide, {1: L.LACACHE_STAGE1_STREAM, 2: L.LACACHE_STAGE1_STREAM, 3: L.LACACHE_STAGE1_TENSOR})):
        st = oracle_store(w)
        with new_cache(w, L.LACACHE_STAGE1_AUTO) as cache:
            fill(cache, w)
            full = wl.batch(w, 0, device="cuda")
            for B, kernel in want.items():
                q = {k: full[k][:B].contiguous() for k in ("emb", "prefix", "ids")}
                g = gpu_lookup(cache, q)
                assert cache.last_launch()[1] == kernel, (w.n, B)
                p = params(w)
                oq = oracle_queries(q)
                rep = compare(g, oracle.lookup(st, oq, p), p, pair_scores=pair_scores_fn(st, oq))
                assert rep.exact + rep.band == B


@pytest.mark.parametrize("stage1", PATHS)
def test_odd_number_of_query_tiles(stage1):
    # B = 300: three query tiles; the tensor kernel pairs query tiles on two-CTA clusters, so the third tile's
    # partner has no queries. n = 12,050: the last key tile holds 18 keys, so its upper half (the second CTA's
    # box) has none either.
    w = wl.WORKLOADS["serve-2m"].scaled(n=12_050, batch=300, clusters=120)
    rep = run_parity(w, stage1)
    assert rep.exact + rep.band == w.batch and rep.band <= 2


@pytest.mark.parametrize("stage1", PATHS)
@pytest.mark.parametrize("mode,tmin", [(oracle.CHECK_TOKENS, None), (oracle.CHECK_TOKENS, 2),
                                       (oracle.CHECK_BOTH, None), (oracle.CHECK_BOTH, 3)])
def test_check_modes(stage1, mode, tmin):
    w = wl.WORKLOADS["tiny-4k"].scaled(n=3000, k=4, vocab=3, batch=48)   # small vocab: partial token matches
    rep = run_parity(w, stage1, check_mode=mode, token_match_min=tmin)
    assert rep.exact + rep.band == w.batch


@pytest.mark.parametrize("stage1", PATHS)
@pytest.mark.parametrize("top_c", [1, 32])
def test_top_c_extremes(stage1, top_c):
    w = wl.WORKLOADS["tiny-4k"].scaled(top_c=top_c, batch=40)
    rep = run_parity(w, stage1)
    assert rep.exact + rep.band == w.batch


@pytest.mark.parametrize("stage1", PATHS)
def test_ensemble_of_lookahead_checks(stage1):
    """Three lookahead checks (1024-, 384- and 768-dim prefix embeddings): a hit needs all three (section 3.4)."""
    w = wl.WORKLOADS["ensemble-1m"].scaled(n=70_000, batch=48)
    rep = run_parity(w, stage1)
    assert rep.exact + rep.band == w.batch and rep.band <= 1
    assert rep.hits > 0 and rep.rejects > 0


def test_ensemble_full_size_rejects_prefix_mimics():
    """ensemble-1m at full size (1,048,576 entries): every query checked; the collisions whose prefix matches the
    victim's under the first model only are rejected by the ensemble."""
    w = wl.WORKLOADS["ensemble-1m"]
    st = oracle_store(w)
    with new_cache(w, L.LACACHE_STAGE1_TENSOR) as cache:
        fill(cache, w)
        q = wl.batch(w, 0, device="cuda")
        g = gpu_lookup(cache, q)
    assert g["prefix_scores"].shape == (w.batch, 3)
    oq = oracle_queries(q)
    p = params(w)
    rep = compare(g, oracle.lookup(st, oq, p), p, pair_scores=pair_scores_fn(st, oq))
    log_report(f"{w.name} full size", rep)
    assert rep.exact + rep.band == w.batch and rep.band <= 1
    cls = q["class"].numpy()
    assert np.all(g["status"][cls == wl.MIMIC] == L.LACACHE_REJECT)
    assert np.all(g["status"][cls == wl.NEAR] == L.LACACHE_HIT)


def _dev(a, dtype=torch.bfloat16):
    return torch.tensor(np.asarray(a, np.float32), device="cuda").to(dtype).contiguous()


@pytest.mark.parametrize("stage1", PATHS)
def test_hand_built_duplicates_thresholds_and_order(stage1):
    d = 64
    e = np.eye(d)
    half = np.zeros(d)
    half[:4] = 0.5
    keys = np.stack([e[1], e[0], e[0], half, e[0]])          # entries 1, 2, 4 share a key
    pres = np.stack([e[5], e[6], e[7], e[8], e[7]])
    ids = np.array([[1, 1], [2, 2], [3, 3], [4, 4], [3, 3]], np.int32)
    qs = np.stack([e[0], e[0], half, e[9], e[0]])
    qp = np.stack([e[7], e[6], e[8], e[9], e[5]])
    qi = np.array([[3, 3], [2, 2], [4, 4], [0, 0], [0, 0]], np.int32)
    # tau_c = 0.5: query 2 (= half) scores exactly 0.5 against entry 3 and entries 1, 2, 4 (inclusive)
    with L.LaCache(d, 2, 16, 0.5, 0.5, 4, max_batch=8, stage1=stage1) as c:
        c.insert(_dev(keys), _dev(pres), torch.tensor(ids, device="cuda"))
        out = c.lookup(_dev(qs), _dev(qp), torch.tensor(qi, device="cuda"))
        torch.cuda.synchronize()
        g = {k: v.cpu().numpy() for k, v in out.items()}
    assert list(g["status"]) == [L.LACACHE_HIT, L.LACACHE_HIT, L.LACACHE_HIT, L.LACACHE_MISS_KEY,
                                 L.LACACHE_REJECT]
    # query 0: candidates 1, 2, 4 tie at 1.0 -> id order; entry 1's prefix e6 fails, entry 2's e7 passes
    assert list(g["cand_id"][0]) == [1, 2, 4, 3] and g["entry_id"][0] == 2
    assert np.all(g["cand_score"][0, :3] == 1.0) and g["cand_score"][0, 3] == 0.5
    assert g["entry_id"][1] == 1 and g["token_matches"][1] == 2
    assert g["entry_id"][2] == 3 and g["key_score"][2] == 1.0
    assert g["n_cand"][3] == 0 and g["key_score"][3] == 0.0 and np.isnan(g["prefix_score"][3])
    assert g["entry_id"][4] == -1 and g["prefix_score"][4] == 0.0 and g["token_matches"][4] == 0


@pytest.mark.parametrize("stage1", PATHS)
@pytest.mark.parametrize("tau_c", [0.0, -0.25])
def test_signed_zero_scores_tie_by_id(stage1, tau_c):
    """Scores of +0.0 and -0.0 are equal: at a key threshold <= 0 every entry below is a candidate, and the tie
    goes to the lower id whatever the zero's sign. Even entries are all +0.0, odd ones all -0.0, so every product
    of a query with an odd entry is a negative zero."""
    d, n = 64, 12
    keys = np.zeros((n, d))
    keys[1::2] = -0.0
    pres = np.tile(np.eye(d)[1], (n, 1))
    ids = np.zeros((n, 2), np.int32)
    e = np.eye(d)
    qs = np.stack([e[0], -e[0], e[3]])
    with L.LaCache(d, 2, 16, tau_c, -1.0, 4, max_batch=8, stage1=stage1) as c:
        c.insert(_dev(keys), _dev(pres), torch.tensor(ids, device="cuda"))
        out = c.lookup(_dev(qs), _dev(qs), torch.zeros((3, 2), dtype=torch.int32, device="cuda"))
        torch.cuda.synchronize()
        g = {k: v.cpu().numpy() for k, v in out.items()}
    for b in range(3):
        assert list(g["cand_id"][b]) == [0, 1, 2, 3], (b, g["cand_id"][b])
        assert np.all(g["cand_score"][b] == 0.0) and g["n_cand"][b] == 4
        assert g["status"][b] == L.LACACHE_HIT and g["entry_id"][b] == 0


@pytest.mark.parametrize("stage1", PATHS)
def test_empty_cache_is_all_key_misses(stage1):
    with L.LaCache(64, 4, 128, 0.9, 0.8, 4, max_batch=8, stage1=stage1) as c:
        q = _dev(np.eye(64)[:3])
        out = c.lookup(q, q, torch.zeros((3, 4), dtype=torch.int32, device="cuda"))
        torch.cuda.synchronize()
        assert torch.all(out["status"] == L.LACACHE_MISS_KEY)
        assert torch.all(out["key_score"] == -math.inf) and torch.all(out["entry_id"] == -1)
        assert torch.all(out["cand_id"] == -1) and c.last_launch()[0] == 0


@pytest.mark.parametrize("stage1", PATHS)
def test_host_buffer_lookup_matches_device_lookup(stage1):
    w = wl.WORKLOADS["tiny-4k"]
    with new_cache(w, stage1) as cache:
        fill(cache, w)
        q = wl.batch(w, 0, device="cuda")
        g = gpu_lookup(cache, q)
        hq = {k: q[k].cpu().pin_memory() for k in ("emb", "prefix", "ids")}
        out = L.alloc_result(w.batch, w.top_c, "cpu", pinned=True)
        L.lacache_lookup_host(cache.h, hq["emb"], hq["prefix"], hq["ids"], out)
        for k, v in out.items():
            assert np.array_equal(v.numpy(), g[k], equal_nan=True), k


def _host_copy(t, kind, offset=0):
    """A host copy of tensor t: pinned, pageable, or pinned at `offset` bytes past a 16-byte boundary."""
    if kind == "pageable":
        return t.cpu().clone()
    raw = torch.empty(t.numel() * t.element_size() + offset, dtype=torch.uint8).pin_memory()
    v = raw[offset:].view(t.dtype).view(t.shape)
    v.copy_(t.cpu())
    return v


@pytest.mark.parametrize("kinds", [("pageable", "pageable", "pageable"), ("pinned+2", "pinned+6", "pinned+4"),
                                   ("pinned", "pageable", "pinned+4")], ids=["pageable", "misaligned", "mixed"])
def test_host_buffer_lookup_any_host_memory(kinds):
    # inputs in mapped pinned memory are gathered by a kernel, others copied by DMA; results written to the
    # library's mapped staging are copied into any host arrays. B = 300 also covers the CTA-pair kernel.
    w = wl.WORKLOADS["serve-2m"].scaled(n=12_050, batch=300, clusters=120)
    with new_cache(w, L.LACACHE_STAGE1_TENSOR) as cache:
        fill(cache, w)
        q = wl.batch(w, 0, device="cuda")
        g = gpu_lookup(cache, q)
        hq = {}
        for key, kind in zip(("emb", "prefix", "ids"), kinds):
            off = int(kind.split("+")[1]) if "+" in kind else 0
            hq[key] = _host_copy(q[key], "pageable" if kind == "pageable" else "pinned", off)
            assert (hq[key].data_ptr() % 16 == 0) == (off == 0)
        out = L.alloc_result(w.batch, w.top_c, "cpu", pinned=kinds[0] != "pageable")
        for _ in range(2):   # twice: the second call reuses the staging
            L.lacache_lookup_host(cache.h, hq["emb"], hq["prefix"], hq["ids"], out)
            for k, v in out.items():
                assert np.array_equal(v.numpy(), g[k], equal_nan=True), k
        assert cache.last_launch()[1] == L.LACACHE_STAGE1_TENSOR_PAIR


@pytest.mark.parametrize("stage1", PATHS)
def test_async_host_lookups_in_flight_match_device_lookups(stage1):
    # three lookups enqueued back to back on one stream, each into its own mapped pinned outputs, read only after
    # the stream has passed them; the inputs sit in mapped pinned memory, two of them off 16-byte boundaries
    w = wl.WORKLOADS["serve-2m"].scaled(n=12_050, batch=300 if stage1 == L.LACACHE_STAGE1_TENSOR else 64,
                                        clusters=120)
    with new_cache(w, stage1) as cache:
        fill(cache, w)
        qs = [wl.batch(w, i, device="cuda") for i in range(3)]
        want = [gpu_lookup(cache, q) for q in qs]
        hq = [{k: _host_copy(q[k], "pinned", off) for k, off in (("emb", 0), ("prefix", 2), ("ids", 4))}
              for q in qs]
        outs = [L.alloc_result(w.batch, w.top_c, "cpu", pinned=True) for _ in qs]
        stream = torch.cuda.current_stream()
        for q, o in zip(hq, outs):
            L.lacache_lookup_host_async(cache.h, q["emb"], q["prefix"], q["ids"], o, stream)
        stream.synchronize()
        cache.sync()
        for o, g in zip(outs, want):
            for k, v in o.items():
                assert np.array_equal(v.numpy(), g[k], equal_nan=True), k


def test_host_lookups_interleaved_with_device_lookups_keep_their_inputs():
    # Host lookups stage their inputs in two slots used in turn, and each one's gather may run while the lookup
    # before it is still in stage 2. Eight lookups are enqueued back to back on one stream, host and device
    # lookups mixed, each with its own batch; k = 5 makes a slot's size no multiple of 16 bytes.
    w = wl.WORKLOADS["tiny-4k"].scaled(k=5, batch=48)
    kinds = ["host", "host", "device", "host", "host", "host", "device", "host"]
    with new_cache(w, L.LACACHE_STAGE1_TENSOR) as cache:
        fill(cache, w)
        qs = [wl.batch(w, i, device="cuda") for i in range(len(kinds))]
        want = [gpu_lookup(cache, q) for q in qs]
        stream = torch.cuda.current_stream()
        outs = []
        for kind, q in zip(kinds, qs):
            if kind == "host":
                hq = {k: _host_copy(q[k], "pinned") for k in ("emb", "prefix", "ids")}
                o = L.alloc_result(w.batch, w.top_c, "cpu", pinned=True)
                L.lacache_lookup_host_async(cache.h, hq["emb"], hq["prefix"], hq["ids"], o, stream)
                outs.append((o, hq))
            else:
                outs.append((cache.lookup(q["emb"], q["prefix"], q["ids"], cuda_stream=stream), None))
        stream.synchronize()
        cache.sync()
        for (o, _), g in zip(outs, want):
            for k, v in o.items():
                assert np.array_equal(v.cpu().numpy(), g[k], equal_nan=True), k


def test_async_host_lookup_refuses_unmapped_or_misaligned_buffers():
    w = wl.WORKLOADS["tiny-4k"]
    with new_cache(w, L.LACACHE_STAGE1_TENSOR) as cache:
        fill(cache, w)
        q = wl.batch(w, 0, device="cuda")
        pinned = {k: q[k].cpu().pin_memory() for k in ("emb", "prefix", "ids")}
        pageable = {k: q[k].cpu() for k in ("emb", "prefix", "ids")}
        out = L.alloc_result(w.batch, w.top_c, "cpu", pinned=True)
        for v in out.values():
            v.fill_(7)
        cases = []
        for key in ("emb", "prefix", "ids"):    # one pageable input
            cases.append(({**pinned, key: pageable[key]}, out))
        cases.append((pinned, {**out, "cand_score": torch.empty((w.batch, w.top_c))}))   # a pageable output
        raw = torch.empty(w.batch * 4 + 4, dtype=torch.uint8).pin_memory()
        cases.append((pinned, {**out, "key_score": raw.data_ptr() + 2}))                # a misaligned output
        for qi, o in cases:
            with pytest.raises(L.LacacheError) as e:
                L.lacache_lookup_host_async(cache.h, qi["emb"], qi["prefix"], qi["ids"], o)
            assert e.value.status == L.LACACHE_ERR_INVALID_ARG
        torch.cuda.synchronize()
        for v in out.values():      # nothing ran
            assert torch.all(v == 7)


@pytest.mark.parametrize("stage1", PATHS)
def test_serve_loop_appends_misses_like_the_oracle(stage1):
    w = wl.WORKLOADS["serve-2m"].scaled(n=20_000, batch=64, clusters=200)
    steps = 12
    loop = oracle.ServeLoop(w.n + steps * w.batch, w.d, w.k, params(w))
    st = oracle_store(w)
    loop.insert(st.key, st.prefix, st.ids)
    with new_cache(w, stage1, capacity=w.n + steps * w.batch) as cache:
        fill(cache, w)
        for step in range(steps):
            q = wl.batch(w, step, device="cuda")
            out = cache.lookup(q["emb"], q["prefix"], q["ids"])
            first, m = cache.append_misses(q["emb"], q["prefix"], q["ids"], out["status"])
            g = {k: v.cpu().numpy() for k, v in out.items()}
            oq = oracle_queries(q)
            res, ofirst, om = loop.step(oq)
            rep = compare(g, res, loop.params)
            assert rep.band == 0 and (first, m) == (ofirst, om) and cache.size == loop.n
        # the appended rows are the non-HIT queries, in order, bit for bit
        n = cache.size - w.n
        key = torch.empty((n, w.d), dtype=torch.bfloat16, device="cuda")
        ids = torch.empty((n, w.k), dtype=torch.int32, device="cuda")
        L.lacache_read_rows(cache.h, w.n, n, key=key, ids=ids)
        torch.cuda.synchronize()
        assert np.array_equal(wl.bf16_bits(key), loop.store.key[w.n:loop.n])
        assert np.array_equal(ids.cpu().numpy(), loop.store.ids[w.n:loop.n])


@pytest.mark.parametrize("batch", [32, 200], ids=["dynamic-schedule", "cta-pairs"])
def test_two_handles_look_up_concurrently_on_two_streams(batch):
    # Each handle owns its store, scratch and schedule counters: lookups of two handles interleaved on two streams,
    # several in flight at once, give each handle's own sequential results.
    wa = wl.WORKLOADS["mid-1m"].scaled(n=60_000, batch=batch)
    wb = wl.WORKLOADS["serve-2m"].scaled(n=45_000, batch=batch, clusters=300)
    with new_cache(wa, L.LACACHE_STAGE1_TENSOR) as ca, new_cache(wb, L.LACACHE_STAGE1_TENSOR) as cb:
        fill(ca, wa)
        fill(cb, wb)
        qa = [wl.batch(wa, i, device="cuda") for i in range(3)]
        qb = [wl.batch(wb, i, device="cuda") for i in range(3)]
        want_a = [gpu_lookup(ca, q) for q in qa]
        want_b = [gpu_lookup(cb, q) for q in qb]
        sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
        outs_a = [L.alloc_result(batch, wa.top_c, "cuda") for _ in qa]
        outs_b = [L.alloc_result(batch, wb.top_c, "cuda") for _ in qb]
        torch.cuda.synchronize()
        for _ in range(2):
            for i in range(3):
                ca.lookup(qa[i]["emb"], qa[i]["prefix"], qa[i]["ids"], out=outs_a[i], cuda_stream=sa)
                cb.lookup(qb[i]["emb"], qb[i]["prefix"], qb[i]["ids"], out=outs_b[i], cuda_stream=sb)
        torch.cuda.synchronize()
        ca.sync()
        cb.sync()
        for outs, want in ((outs_a, want_a), (outs_b, want_b)):
            for o, g in zip(outs, want):
                for k, v in o.items():
                    assert np.array_equal(v.cpu().numpy(), g[k], equal_nan=True), k


@pytest.mark.parametrize("stage1", PATHS)
def test_back_to_back_lookups_of_mixed_sizes_match_lookups_run_alone(stage1):
    # A lookup's stage 1 scans while the previous lookup's stage 2 finishes, and both use the handle's partial-list
    # scratch and schedule counters. Lookups of changing batch size (single CTAs on the dynamic schedule and CTA
    # pairs, growing and shrinking the scratch they cover), enqueued back to back with no synchronization, must
    # each give the result of the same lookup run alone.
    w = wl.WORKLOADS["mid-1m"].scaled(n=60_000, batch=200)
    sizes = [32, 7, 200, 64, 1, 130, 32, 200, 5]
    with new_cache(w, stage1) as cache:
        fill(cache, w)
        full = [wl.batch(w, i, device="cuda") for i in range(len(sizes))]
        qs = [{k: full[i][k][:b].contiguous() for k in ("emb", "prefix", "ids")} for i, b in enumerate(sizes)]
        alone = [gpu_lookup(cache, q) for q in qs]
        outs = [L.alloc_result(b, w.top_c, "cuda") for b in sizes]
        torch.cuda.synchronize()
        for rep in range(2):
            for q, o in zip(qs, outs):
                cache.lookup(q["emb"], q["prefix"], q["ids"], out=o)
            torch.cuda.synchronize()
            cache.sync()
            for o, g in zip(outs, alone):
                for k, v in o.items():
                    assert np.array_equal(v.cpu().numpy(), g[k], equal_nan=True), (rep, k)


def test_insert_is_all_or_nothing_on_capacity():
    with L.LaCache(64, 2, 10, 0.9, 0.8, 2, max_batch=4) as c:
        rows = _dev(np.eye(64)[:8])
        ids = torch.zeros((8, 2), dtype=torch.int32, device="cuda")
        assert c.insert(rows, rows, ids) == 0
        with pytest.raises(L.LacacheError) as e:
            c.insert(rows, rows, ids)
        assert e.value.status == L.LACACHE_ERR_CAPACITY and c.size == 8
        assert c.insert(rows[:2], rows[:2], ids[:2]) == 8 and c.size == 10


def test_invalid_lookup_arguments():
    with L.LaCache(64, 2, 10, 0.9, 0.8, 2, max_batch=4) as c:
        q = _dev(np.eye(64)[:8])
        ids = torch.zeros((8, 2), dtype=torch.int32, device="cuda")
        with pytest.raises(L.LacacheError) as e:
            c.lookup(q, q, ids)                              # B = 8 > max_batch
        assert e.value.status == L.LACACHE_ERR_INVALID_ARG
        flat = torch.zeros(64 * 4 + 1, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(L.LacacheError):
            c.lookup(flat[1:].view(4, 64), q[:4], ids[:4])    # misaligned embedding pointer


@pytest.mark.parametrize("stage1", PATHS)
def test_mid_cache_full_size(stage1):
    """The benchmark workload at full size: 1,048,576 entries, d = 768, B = 32, every query checked."""
    rep = run_parity(wl.WORKLOADS["mid-1m"], stage1)
    assert rep.exact + rep.band == 32 and rep.band <= 1
    assert rep.hits > 0 and rep.rejects > 0 and rep.misses > 0


def test_decision_counters_match_the_outputs():
    w = wl.WORKLOADS["tiny-4k"]
    with new_cache(w, L.LACACHE_STAGE1_TENSOR, capacity=w.n + 2 * w.batch) as cache:
        fill(cache, w)
        assert cache.stats(reset=True)["inserted"] == w.n
        want = {"hits": 0, "rejects": 0, "key_misses": 0}
        for step in range(3):
            q = wl.batch(w, step, device="cuda")
            out = cache.lookup(q["emb"], q["prefix"], q["ids"])
            st = out["status"].cpu().numpy()
            want["hits"] += int((st == L.LACACHE_HIT).sum())
            want["rejects"] += int((st == L.LACACHE_REJECT).sum())
            want["key_misses"] += int((st == L.LACACHE_MISS_KEY).sum())
        _, appended = cache.append_misses(q["emb"], q["prefix"], q["ids"], out["status"])
        got = cache.stats(reset=True)
        assert got["lookups"] == 3 and got["queries"] == 3 * w.batch and got["inserted"] == 0
        assert {k: got[k] for k in want} == want and got["appended"] == appended
        assert min(want.values()) > 0
        assert cache.stats() == {k: 0 for k in got}


@pytest.mark.parametrize("top_c", [1, 2, 16, 32])
@pytest.mark.parametrize("batch", [40, 200], ids=["single-cta", "cta-pairs"])
def test_candidate_list_sizes(top_c, batch):
    # every epilogue list size of the tensor kernel (4, 8, 16, 32 slots), on one query tile and on CTA pairs;
    # top_c = 1 and 2 also make the candidate cut bind for most near-duplicates and collisions
    w = wl.WORKLOADS["serve-2m"].scaled(n=20_000, batch=batch, clusters=150, top_c=top_c)
    rep = run_parity(w, L.LACACHE_STAGE1_TENSOR)
    assert rep.exact + rep.band == w.batch and rep.band <= 2
    assert rep.hits > 0 and rep.rejects > 0 and rep.misses > 0


@pytest.mark.parametrize("batch", [32, 200], ids=["dynamic-schedule", "cta-pairs"])
@pytest.mark.parametrize("stage1", PATHS)
def test_lookup_captured_in_a_cuda_graph_replays_like_eager_lookups(stage1, batch):
    # the stage-1 schedule keeps no host-side state between launches, so one captured lookup can be replayed
    w = wl.WORKLOADS["mid-1m"].scaled(n=70_000, batch=batch)
    with new_cache(w, stage1) as cache:
        fill(cache, w)
        q0, q1 = wl.batch(w, 0, device="cuda"), wl.batch(w, 1, device="cuda")
        eager = []
        for q in (q0, q1):
            eager.append({k: v.clone() for k, v in cache.lookup(q["emb"], q["prefix"], q["ids"]).items()})
        torch.cuda.synchronize()
        cache.sync()
        inp = {k: q0[k].clone() for k in ("emb", "prefix", "ids")}
        out = L.alloc_result(w.batch, w.top_c, "cuda")
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):                 # warm-up on the capture stream, as torch asks
            L.lacache_lookup(cache.h, inp["emb"], inp["prefix"], inp["ids"], out, side)
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, capture_error_mode="relaxed"):
            L.lacache_lookup(cache.h, inp["emb"], inp["prefix"], inp["ids"], out)
        for step, want in ((0, eager[0]), (0, eager[0]), (1, eager[1]), (0, eager[0])):
            src = q0 if step == 0 else q1
            for k in inp:
                inp[k].copy_(src[k])
            graph.replay()
            torch.cuda.synchronize()
            cache.sync()
            for k in out:
                assert torch.equal(out[k].view(torch.uint8), want[k].view(torch.uint8)), (step, k)
