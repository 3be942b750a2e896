"""Save and load of a cache: the loaded handle has the saved configuration and entries, looks up bit for bit as
the saved one did, keeps entry ids, and accepts appends up to its new capacity."""
import pytest
import torch

from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl
from parity import fill, new_cache

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


@pytest.mark.parametrize("name", ["tiny-4k", "ensemble-1m"])
def test_saved_cache_loads_and_looks_up_identically(name, tmp_path):
    w = wl.WORKLOADS[name].scaled(n=5_000, batch=48) if name != "tiny-4k" else wl.WORKLOADS[name]
    path = str(tmp_path / "cache.lacache")
    q = wl.batch(w, 0, device="cuda")
    with new_cache(w, L.LACACHE_STAGE1_TENSOR) as cache:
        fill(cache, w)
        before = {k: v.clone() for k, v in cache.lookup(q["emb"], q["prefix"], q["ids"]).items()}
        cache.sync()
        cache.save(path)
        saved_cfg, saved_ens = L.lacache_get_config(cache.h)
    with pytest.raises(L.LacacheError) as e:
        L.LaCache.load(path, capacity=w.n - 1)
    assert e.value.status == L.LACACHE_ERR_CAPACITY
    loaded = L.LaCache.load(path, capacity=w.n + w.batch)
    try:
        cfg, ens = L.lacache_get_config(loaded.h)
        assert cfg.capacity == w.n + w.batch and cfg.d == saved_cfg.d and cfg.top_c == saved_cfg.top_c
        assert ens.m == saved_ens.m and list(ens.dims) == list(saved_ens.dims)
        assert loaded.size == w.n
        after = loaded.lookup(q["emb"], q["prefix"], q["ids"])
        loaded.sync()
        for k in before:
            assert torch.equal(before[k].view(torch.uint8), after[k].view(torch.uint8)), k
        first, m = loaded.append_misses(q["emb"], q["prefix"], q["ids"], after["status"])
        assert first == w.n and m == int((after["status"] != L.LACACHE_HIT).sum())
    finally:
        loaded.close()


def test_saved_simhash_cache_takes_its_index_again(tmp_path):
    # the index is not saved: the loaded handle (still configured for the SimHash stage) refuses lookups until
    # lacache_enable_lsh signs its entries again, then looks up as the saved one did, appends included
    w = wl.WORKLOADS["mid-1m"].scaled(n=20_000, batch=16)
    bits = 256
    radius = wl.lsh_radius(w.tau_c, bits)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    path = str(tmp_path / "cache.lacache")
    q = wl.batch(w, 0, device="cuda")
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        L.lacache_enable_lsh(cache.h, bits, radius, R)
        before = {k: v.clone() for k, v in cache.lookup(q["emb"], q["prefix"], q["ids"]).items()}
        cache.sync()
        cache.save(path)
    loaded = L.LaCache.load(path, capacity=w.n + w.batch)
    try:
        with pytest.raises(L.LacacheError) as e:
            loaded.lookup(q["emb"], q["prefix"], q["ids"])
        assert e.value.status == L.LACACHE_ERR_INVALID_ARG
        L.lacache_enable_lsh(loaded.h, bits, radius, R)
        after = loaded.lookup(q["emb"], q["prefix"], q["ids"])
        loaded.sync()
        assert loaded.last_launch()[1] == L.LACACHE_STAGE1_LSH
        for k in before:
            assert torch.equal(before[k].view(torch.uint8), after[k].view(torch.uint8)), k
        first, m = loaded.append_misses(q["emb"], q["prefix"], q["ids"], after["status"])
        again = loaded.lookup(q["emb"], q["prefix"], q["ids"])
        loaded.sync()
        # every appended query now finds its own row (an exact copy) through the index
        miss = torch.nonzero(after["status"] != L.LACACHE_HIT).flatten()
        assert m == len(miss)
        got = again["cand_id"][miss]
        want = torch.arange(first, first + m, device="cuda", dtype=got.dtype)
        assert torch.all((got == want[:, None]).any(dim=1))
    finally:
        loaded.close()
