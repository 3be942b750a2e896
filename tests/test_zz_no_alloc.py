"""lacache_lookup_noalloc: the lookup for callers that cannot allocate device memory.

Callers under a runtime or framework allocator that owns all device memory, or that must not trigger the
synchronization cudaMalloc/cudaFree can cause, cannot create a handle (lacache_create allocates the store and the
stage-1 scratch). This entry point takes the cache rows as the caller's device arrays and keeps its scratch in a
fixed device array of the library. The test checks it against lacache_lookup on the same rows, two calls in a
row, and that a batch too large for the fixed scratch is refused. This file is named so pytest collects it last.
"""
import numpy as np
import pytest
import torch

from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

TOL = 2e-3


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


def _rows(w):
    keys, pres, ids = [], [], []
    for ch in wl.iter_store(w, "cuda"):
        keys.append(ch["key"])
        pres.append(ch["prefix"])
        ids.append(ch["ids"])
    return torch.cat(keys).contiguous(), torch.cat(pres).contiguous(), torch.cat(ids).contiguous()


def _same(a: dict, b: dict):
    for name in ("status", "entry_id", "n_cand", "token_matches", "cand_id", "cand_matches"):
        assert torch.equal(a[name], b[name]), name
    for name in ("key_score", "prefix_score", "cand_score", "cand_prefix_score"):
        x, y = a[name].cpu().numpy(), b[name].cpu().numpy()
        both_nan = np.isnan(x) & np.isnan(y)
        assert np.all(both_nan | (np.abs(x - y) <= TOL) | (x == y)), name


@pytest.mark.parametrize("batch", [96, 256], ids=["one-tile", "cta-pairs"])
@pytest.mark.parametrize("stage1", [L.LACACHE_STAGE1_TENSOR, L.LACACHE_STAGE1_STREAM], ids=["tensor", "stream"])
def test_noalloc_lookup_matches_the_handle_lookup(stage1, batch):
    w = wl.WORKLOADS["mid-1m"].scaled(n=50_000, batch=batch)
    key, pre, ids = _rows(w)
    with L.LaCache(w.d, w.k, w.n, w.tau_c, w.tau_a, w.top_c, max_batch=w.batch, stage1=stage1) as cache:
        cache.insert(key, pre, ids)
        for step in (0, 1):                       # two calls in a row share the fixed scratch
            q = wl.batch(w, step, device="cuda")
            ref = cache.lookup(q["emb"], q["prefix"], q["ids"])
            out = L.alloc_result(w.batch, w.top_c, "cuda")
            L.lacache_lookup_noalloc(cache.cfg, key, pre, ids, q["emb"], q["prefix"], q["ids"], out)
            torch.cuda.synchronize()
            _same(out, ref)
            assert int((out["status"] == L.LACACHE_HIT).sum()) > 0


@pytest.mark.parametrize("mode,tmin,top_c,stage1", [
    (L.LACACHE_CHECK_TOKENS, 12, 8, L.LACACHE_STAGE1_TENSOR),
    (L.LACACHE_CHECK_BOTH, 12, 8, L.LACACHE_STAGE1_STREAM),
    (L.LACACHE_CHECK_EMB, 0, 1, L.LACACHE_STAGE1_AUTO),
    (L.LACACHE_CHECK_EMB, 0, 32, L.LACACHE_STAGE1_AUTO),
    (L.LACACHE_CHECK_TOKENS, 12, 32, L.LACACHE_STAGE1_STREAM),
], ids=["tokens-12", "both-12", "top1-auto", "top32-auto", "tokens-top32-stream"])
def test_noalloc_modes_and_list_sizes(mode, tmin, top_c, stage1):
    """The check modes with a partial token match, the smallest and largest candidate lists, and AUTO: each filled
    into stage 2's arguments by the no-alloc entry point itself, against the handle's lookup."""
    w = wl.WORKLOADS["mid-1m"].scaled(n=30_000, batch=64, top_c=top_c)
    key, pre, ids = _rows(w)
    with L.LaCache(w.d, w.k, w.n, w.tau_c, w.tau_a, w.top_c, max_batch=w.batch, stage1=stage1, check_mode=mode,
                   token_match_min=tmin) as cache:
        cache.insert(key, pre, ids)
        for step in (0, 1):
            q = wl.batch(w, step, device="cuda")
            ref = cache.lookup(q["emb"], q["prefix"], q["ids"])
            out = L.alloc_result(w.batch, w.top_c, "cuda")
            L.lacache_lookup_noalloc(cache.cfg, key, pre, ids, q["emb"], q["prefix"], q["ids"], out)
            torch.cuda.synchronize()
            _same(out, ref)


def test_noalloc_auto_on_a_small_store_takes_the_streaming_scan():
    """AUTO chooses as for a handle: two queries against 15 MB of keys take the streaming scan, in both entry
    points, and give the same results."""
    w = wl.WORKLOADS["mid-1m"].scaled(n=10_000, batch=2)
    key, pre, ids = _rows(w)
    with L.LaCache(w.d, w.k, w.n, w.tau_c, w.tau_a, w.top_c, max_batch=w.batch) as cache:
        cache.insert(key, pre, ids)
        for step in (0, 1):
            q = wl.batch(w, step, device="cuda")
            ref = cache.lookup(q["emb"], q["prefix"], q["ids"])
            assert cache.last_launch()[1] == L.LACACHE_STAGE1_STREAM
            out = L.alloc_result(w.batch, w.top_c, "cuda")
            L.lacache_lookup_noalloc(cache.cfg, key, pre, ids, q["emb"], q["prefix"], q["ids"], out)
            torch.cuda.synchronize()
            _same(out, ref)


def _empty_batch(B, d, k):
    g = torch.Generator(device="cuda").manual_seed(B)
    q = torch.randn((B, d), generator=g, device="cuda").to(torch.bfloat16)
    qi = torch.randint(0, 100, (B, k), generator=g, device="cuda", dtype=torch.int32)
    return q, qi


def test_noalloc_empty_cache_and_largest_batch():
    """With no rows (n = 0) stage 1 does not run and stage 2 sees no partial list: every query is a key miss, as
    for an empty handle. The batch is the largest the fixed scratch takes at top_c = 32:
    B * (8 * top_c + 8) <= 8 MiB - 512 bytes."""
    d, k, top_c = 64, 4, 32
    B = ((8 << 20) - 512) // (8 * top_c + 8)
    q, qi = _empty_batch(B, d, k)
    cfg = L.make_config(d, k, 1, 0.9, 0.8, top_c, max_batch=B)
    for _ in range(2):
        out = L.alloc_result(B, top_c, "cuda")
        L.lacache_lookup_noalloc(cfg, None, None, None, q, q, qi, out)
        torch.cuda.synchronize()
        assert torch.all(out["status"] == L.LACACHE_MISS_KEY)
        assert torch.all(out["entry_id"] == -1) and torch.all(out["n_cand"] == 0)
        assert torch.all(torch.isneginf(out["key_score"])) and torch.all(torch.isnan(out["prefix_score"]))
        assert torch.all(out["cand_id"] == -1)
    with L.LaCache(d, k, 1, 0.9, 0.8, top_c, max_batch=256) as cache:
        ref = cache.lookup(q[:256], q[:256], qi[:256])
        torch.cuda.synchronize()
    _same({name: v[:256] for name, v in out.items()}, ref)


def test_noalloc_refuses_a_batch_larger_than_its_scratch():
    d, top_c = 64, 32
    cfg = L.make_config(d, 4, 1, 0.9, 0.8, top_c, max_batch=1)
    B = ((8 << 20) - 512) // (8 * top_c + 8) + 1    # one query more than fits the 8 MiB scratch
    q = torch.zeros((B, d), dtype=torch.bfloat16, device="cuda")
    qi = torch.zeros((B, 4), dtype=torch.int32, device="cuda")
    out = L.alloc_result(B, top_c, "cuda", candidates=False)
    with pytest.raises(L.LacacheError) as e:
        L.lacache_lookup_noalloc(cfg, None, None, None, q, q, qi, out)
    assert e.value.status == L.LACACHE_ERR_UNSUPPORTED
