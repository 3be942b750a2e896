"""Parity of the SimHash-indexed lookup on seeded random configurations: each case draws the signature width, the
radius (the one the threshold gives, or any from 0 to the whole signature), the batch size (across the popcount
scan's passes and the switch to the tensor-core scan), the store size, d, top_c and the threshold, and compares
the lookup through the C ABI with the oracle's SimHash lookup on the same bytes. Queries whose outcome an ambiguous
signature bit could change are set aside (at most 1 in 50, and at most 2)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_01718_gb300 import build
from paper_2608_01718_gb300 import lacache as L
from paper_2608_01718_gb300 import workloads as wl

from parity import compare, fill, gpu_lookup, log_report, new_cache, oracle_queries, oracle_store, params

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def library():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build.build()
    L.load()


def _draw(seed):
    rng = np.random.default_rng(20261203 + seed)
    bits = int(rng.choice([128, 256, 512]))
    d = int(rng.choice([64, 256, 768]))
    tau_c = float(rng.choice([0.8, 0.85, 0.9, 0.95]))
    batch = int(rng.choice([1, 3, 8, 33, 40, 47, 48, 64, 130]))
    n = int(rng.choice([1, 513, 7000, 40_000]))
    top_c = int(rng.choice([1, 4, 8, 32]))
    w = wl.WORKLOADS["mid-1m"].scaled(n=n, d=d, batch=batch, top_c=top_c, tau_c=tau_c, clusters=int(rng.choice([8, 64, 500])))
    radius = wl.lsh_radius(tau_c, bits) if rng.random() < 0.5 else int(rng.integers(0, bits + 1))
    return w, bits, radius


@pytest.mark.parametrize("seed", range(24))
def test_random_simhash_configuration_matches_the_oracle(seed):
    w, bits, radius = _draw(seed)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    st = oracle_store(w)
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        L.lacache_enable_lsh(cache.h, bits, radius, R)
        q = wl.batch(w, 0, device="cuda")
        g = gpu_lookup(cache, q)
        assert cache.last_launch()[1] in (L.LACACHE_STAGE1_LSH, L.LACACHE_STAGE1_LSH_TENSOR)
    p = params(w)
    res, amb = oracle.lookup_lsh(st, oracle_queries(q), p, wl.bf16_bits(R), radius)
    keep = np.nonzero(~amb)[0]
    sub = oracle.Result(**{f: getattr(res, f)[keep] for f in res.__dataclass_fields__})
    rep = compare(g, sub, p, rows=keep)
    log_report(f"random simhash seed={seed} n={w.n} d={w.d} B={w.batch} c={w.top_c} bits={bits} radius={radius} "
               f"tau_c={w.tau_c} ({w.batch - len(keep)} ambiguous)", rep)
    assert len(keep) >= w.batch - min(2, max(1, w.batch // 50))
    assert rep.exact + rep.band == len(keep)
