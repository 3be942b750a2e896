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
