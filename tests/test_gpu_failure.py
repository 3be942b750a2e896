"""Failure detection on the GPU without a fault: a stage-1 wait that runs out is reported, not hung.

lacache_inject_stall makes the tensor kernel's first CTA withhold one TMA load (no copy is issued). The MMA
issuer's bounded wait then runs out (about a second). The kernel records the timeout in the status word, drains
and exits, and lacache_sync reports LACACHE_ERR_DEVICE_TIMEOUT. The context must stay usable: the next lookup
matches the one taken before the injection. With B = 256 the batch runs on CTA pairs: the withholding CTA is the
leader of the first pair, whose abort also stops its peer; both CTAs still meet at the cluster barrier before
freeing the pair's TMEM.

The SimHash popcount scan's ring form (always taken at 512 bits) has the same test: its first CTA withholds the
bulk copy of its first tile, every thread's bounded wait for it runs out, and the CTA ends its pass, waits (bounded)
for the copies it did issue, and exits.
"""
import pytest
import torch

from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


@pytest.mark.parametrize("batch", [32, 256], ids=["single-cta", "cta-pairs"])
def test_stage1_wait_timeout_is_reported_and_the_context_stays_usable(batch):
    # A single query tile runs on the dynamic schedule, where CTAs claim key tiles as they start: with about one
    # tile per CTA a late-starting CTA 0 could claim none and have no load to withhold. 400,000 entries are
    # 1,563 tiles, so CTA 0 always claims some.
    w = wl.WORKLOADS["mid-1m"].scaled(n=400_000 if batch <= 128 else 40_000, batch=batch)
    with L.LaCache(w.d, w.k, w.n, w.tau_c, w.tau_a, w.top_c, max_batch=w.batch,
                   stage1=L.LACACHE_STAGE1_TENSOR) as cache:
        for ch in wl.iter_store(w, "cuda"):
            cache.insert(ch["key"], ch["prefix"], ch["ids"])
        q = wl.batch(w, 0, device="cuda")
        before = {k: v.clone() for k, v in cache.lookup(q["emb"], q["prefix"], q["ids"]).items()}
        cache.sync()
        L.lacache_inject_stall(cache.h, 1)
        cache.lookup(q["emb"], q["prefix"], q["ids"])
        assert cache.last_launch()[1] == (L.LACACHE_STAGE1_TENSOR_PAIR if batch > 128 else L.LACACHE_STAGE1_TENSOR)
        with pytest.raises(L.LacacheError) as e:
            cache.sync()
        assert e.value.status == L.LACACHE_ERR_DEVICE_TIMEOUT
        cache.sync()                                   # the status word was cleared
        after = cache.lookup(q["emb"], q["prefix"], q["ids"])
        cache.sync()
        for k in ("status", "entry_id", "cand_id", "n_cand"):
            assert torch.equal(after[k], before[k]), k


def test_simhash_ring_wait_timeout_is_reported_and_the_context_stays_usable():
    w = wl.WORKLOADS["mid-1m"].scaled(n=40_000, batch=8)
    bits = 512
    with L.LaCache(w.d, w.k, w.n, w.tau_c, w.tau_a, w.top_c, max_batch=w.batch,
                   stage1=L.LACACHE_STAGE1_LSH) as cache:
        for ch in wl.iter_store(w, "cuda"):
            cache.insert(ch["key"], ch["prefix"], ch["ids"])
        L.lacache_enable_lsh(cache.h, bits, wl.lsh_radius(w.tau_c, bits), wl.hyperplanes(bits, w.d, device="cuda"))
        q = wl.batch(w, 0, device="cuda")
        before = {k: v.clone() for k, v in cache.lookup(q["emb"], q["prefix"], q["ids"]).items()}
        cache.sync()
        L.lacache_inject_stall(cache.h, 1)
        cache.lookup(q["emb"], q["prefix"], q["ids"])
        assert cache.last_launch()[1] == L.LACACHE_STAGE1_LSH
        with pytest.raises(L.LacacheError) as e:
            cache.sync()
        assert e.value.status == L.LACACHE_ERR_DEVICE_TIMEOUT
        cache.sync()
        after = cache.lookup(q["emb"], q["prefix"], q["ids"])
        cache.sync()
        for k in ("status", "entry_id", "cand_id", "n_cand"):
            assert torch.equal(after[k], before[k]), k
        # the injection was taken by that lookup: the next one runs clean
        cache.lookup(q["emb"], q["prefix"], q["ids"])
        cache.sync()
