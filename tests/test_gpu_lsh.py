"""GPU parity of the SimHash-indexed key check (Eq. 1; Algorithm 1's cache search) against the oracle.

Signatures are sign decisions of fp32 tensor-core dot products; the oracle takes them in fp64. Bits whose
projection is within 1e-4 of zero may legitimately differ: they are counted, and the queries whose outcome such
a bit could change are excluded from the exact comparison (reported, at most a few)."""
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


def _unpack(words, bits):
    w = words.astype(np.uint64)
    out = np.zeros((w.shape[0], bits), dtype=bool)
    for i in range(bits):
        out[:, i] = (w[:, i // 32] >> np.uint64(i % 32)) & np.uint64(1)
    return out


@pytest.mark.parametrize("bits", [128, 256, 512])
def test_signatures_match_the_oracle(bits):
    w = wl.WORKLOADS["mid-1m"].scaled(n=20_000)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    st = oracle_store(w)
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        L.lacache_enable_lsh(cache.h, bits, 40, R)
        sig = torch.empty((w.n, bits // 32), dtype=torch.int32, device="cuda")
        L.lacache_read_signatures(cache.h, 0, w.n, sig)
        torch.cuda.synchronize()
    got = _unpack(sig.cpu().numpy().view(np.uint32), bits)
    want, amb = oracle.signatures(st.key, wl.bf16_bits(R))
    diff = got != want
    assert not np.any(diff & ~amb), "a signature bit differs away from a zero projection"
    assert amb.mean() < 1e-3


def _expected_lsh_kernel(batch, bits):
    # the tensor-core scan from 48 queries at 256 bits and from 40 at 128 and 512 bits
    return L.LACACHE_STAGE1_LSH_TENSOR if batch >= (48 if bits == 256 else 40) else L.LACACHE_STAGE1_LSH


# popcount-1 / -2: a pass of fewer queries than one group of 8 (only their distances are computed);
# tensor-40: the tensor-core scan at 128 and 512 bits, two passes of the popcount scan at 256 bits (its switch is at
# 48);
# popcount-36: two passes of 32 queries (the handle's max_batch is below the tensor scan's minimum, so it keeps no
# expanded index); tensor-200: two passes of 128 queries at 128 and 256 bits, four of 64 at 512, ragged last pass
@pytest.mark.parametrize("batch", [1, 2, 5, 32, 36, 40, 64, 200],
                         ids=["popcount-1", "popcount-2", "popcount-5", "popcount-32", "popcount-36", "tensor-40",
                              "tensor-64", "tensor-200"])
@pytest.mark.parametrize("bits", [128, 256, 512])
def test_lsh_lookup_matches_the_oracle(bits, batch):
    _check_lsh_lookup(wl.WORKLOADS["mid-1m"].scaled(n=70_000, batch=batch), bits)


@pytest.mark.parametrize("batch", [1, 5])
@pytest.mark.parametrize("bits", [128, 256, 512])
def test_lsh_lookup_at_a_low_threshold_matches_the_oracle(bits, batch):
    # tau_c = 0.8 gives radii of 45, 79 and 142 bits, too wide for the scan's prefix test to reject unrelated
    # pairs: it tests whole signatures (at 512 bits through its shared-memory ring)
    _check_lsh_lookup(wl.WORKLOADS["mid-1m"].scaled(n=70_000, batch=batch, tau_c=0.8), bits)


@pytest.mark.parametrize("bits", [128, 256])
def test_single_query_lookups_on_a_large_store_match_the_oracle(bits):
    # 2.6M entries of d = 64: 304 splits of about 8,553 entries (17 tiles, the last one ragged). One-query lookups
    # on splits of at least 16 tiles stream the signatures through the scan's shared-memory ring (at 512 bits every
    # lookup does, and the cases above cover it); eight such lookups, compared as one batch
    _check_lsh_lookup(wl.WORKLOADS["mid-1m"].scaled(n=2_600_000, d=64, batch=8), bits, one_at_a_time=True)


@pytest.mark.slow
@pytest.mark.parametrize("bits", [128, 256, 512])
def test_lsh_lookup_at_full_size_matches_the_oracle(bits):
    # mid-1m at full size (1,048,576 entries, B = 32), as the benchmark's SimHash line times it: the popcount scan
    # with its prefix test, in its register form at 128 and 256 bits and its shared-memory ring form at 512
    _check_lsh_lookup(wl.WORKLOADS["mid-1m"], bits)


@pytest.mark.parametrize("top_c", [1, 32])
@pytest.mark.parametrize("batch", [16, 64], ids=["popcount", "tensor"])
def test_lsh_top_c_extremes_match_the_oracle(batch, top_c):
    # one candidate per query (every list insertion replaces the head) and the longest lists the kernels hold
    _check_lsh_lookup(wl.WORKLOADS["mid-1m"].scaled(n=40_000, batch=batch, top_c=top_c), 256)


def _check_lsh_lookup(w, bits, one_at_a_time=False):
    batch = w.batch
    radius = wl.lsh_radius(w.tau_c, bits)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    st = oracle_store(w)
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        L.lacache_enable_lsh(cache.h, bits, radius, R)
        q = wl.batch(w, 0, device="cuda")
        if one_at_a_time:
            parts = []
            for i in range(batch):
                parts.append(gpu_lookup(cache, {k: q[k][i:i + 1] for k in ("emb", "prefix", "ids")}))
                assert cache.last_launch()[1] == L.LACACHE_STAGE1_LSH
            g = {k: np.concatenate([r[k] for r in parts]) for k in parts[0]}
        else:
            g = gpu_lookup(cache, q)
            assert cache.last_launch()[1] == _expected_lsh_kernel(batch, bits)
    oq = oracle_queries(q)
    p = params(w)
    res, amb = oracle.lookup_lsh(st, oq, p, wl.bf16_bits(R), radius)
    keep = np.nonzero(~amb)[0]
    sub = oracle.Result(**{f: getattr(res, f)[keep] for f in res.__dataclass_fields__})
    rep = compare(g, sub, p, rows=keep)
    amb_n = w.batch - len(keep)
    log_report(f"lsh bits={bits} B={batch} c={w.top_c} radius={radius} ({amb_n} queries with ambiguous bits)", rep)
    # queries with a signature bit within the fp32/fp64 ambiguity of zero are set aside: at most 1 in 50
    assert rep.exact + rep.band == len(keep) and len(keep) >= w.batch - max(2, w.batch // 50)
    if batch >= 16:
        assert rep.hits > 0 and rep.rejects > 0 and rep.misses > 0
    # at this radius the index keeps every near-duplicate's target: the decisions equal the exact lookup's
    exact = oracle.lookup(st, oq, p)
    assert np.array_equal(res.status, exact.status) and np.array_equal(res.entry_id, exact.entry_id)


@pytest.mark.parametrize("bits", [256, 512])
@pytest.mark.parametrize("batch", [16, 64], ids=["popcount", "tensor"])
def test_full_radius_equals_the_exact_scan_and_appends_are_signed(batch, bits):
    # radius = bits admits every pair: the queue overflows on every tile (at 512 bits the popcount scan's ring form,
    # whose queue is a quarter of the register form's), and appended entries must be signed (in both the packed
    # and the expanded form) before the next lookup
    w = wl.WORKLOADS["serve-2m"].scaled(n=30_000, batch=batch, clusters=300)
    R = wl.hyperplanes(bits, w.d, device="cuda")
    with new_cache(w, L.LACACHE_STAGE1_TENSOR, capacity=w.n + 4 * w.batch) as exact_cache, \
            new_cache(w, L.LACACHE_STAGE1_LSH, capacity=w.n + 4 * w.batch) as lsh_cache:
        fill(exact_cache, w)
        fill(lsh_cache, w)
        L.lacache_enable_lsh(lsh_cache.h, bits, bits, R)      # radius = bits: nothing is pruned
        for step in range(3):
            q = wl.batch(w, step, device="cuda")
            a = exact_cache.lookup(q["emb"], q["prefix"], q["ids"])
            b = lsh_cache.lookup(q["emb"], q["prefix"], q["ids"])
            assert lsh_cache.last_launch()[1] == _expected_lsh_kernel(batch, bits)
            assert torch.equal(a["status"], b["status"]) and torch.equal(a["entry_id"], b["entry_id"])
            assert torch.equal(a["cand_id"], b["cand_id"])
            assert torch.allclose(a["cand_score"], b["cand_score"], atol=2e-3, equal_nan=True)
            exact_cache.append_misses(q["emb"], q["prefix"], q["ids"], a["status"])
            first, m = lsh_cache.append_misses(q["emb"], q["prefix"], q["ids"], b["status"])
        sig = torch.empty((m, bits // 32), dtype=torch.int32, device="cuda")
        L.lacache_read_signatures(lsh_cache.h, first, m, sig)
        torch.cuda.synchronize()
        # the appended entries are the last batch's non-HIT queries, in query order
        miss = torch.nonzero(b["status"] != L.LACACHE_HIT).flatten()
        assert len(miss) == m
        rows = wl.bf16_bits(q["emb"][miss])
    want, amb = oracle.signatures(rows, wl.bf16_bits(R))
    assert not np.any((_unpack(sig.cpu().numpy().view(np.uint32), bits) != want) & ~amb)


@pytest.mark.parametrize("batch", [8, 64], ids=["popcount", "tensor"])
def test_host_buffer_lookups_through_the_index_match_device_lookups(batch):
    # inputs from mapped pinned host memory: the gather kernel writes them, the query-signature kernel waits for
    # it before reading, and three lookups are in flight on one stream (each gather runs under the stage 2 before)
    w = wl.WORKLOADS["mid-1m"].scaled(n=40_000, batch=batch)
    bits = 256
    R = wl.hyperplanes(bits, w.d, device="cuda")
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        L.lacache_enable_lsh(cache.h, bits, wl.lsh_radius(w.tau_c, bits), R)
        qs = [wl.batch(w, i, device="cuda") for i in range(3)]
        want = [gpu_lookup(cache, q) for q in qs]
        hq = [{k: q[k].cpu().pin_memory() for k in ("emb", "prefix", "ids")} for q in qs]
        outs = [L.alloc_result(w.batch, w.top_c, "cpu", pinned=True) for _ in qs]
        stream = torch.cuda.current_stream()
        for q, o in zip(hq, outs):
            L.lacache_lookup_host_async(cache.h, q["emb"], q["prefix"], q["ids"], o, stream)
        stream.synchronize()
        cache.sync()
        assert cache.last_launch()[1] == _expected_lsh_kernel(batch, bits)
        for o, g in zip(outs, want):
            for k, v in o.items():
                assert np.array_equal(v.numpy(), g[k], equal_nan=True), k


def test_lookup_before_the_index_is_enabled_is_refused():
    w = wl.WORKLOADS["mid-1m"].scaled(n=5_000, batch=8)
    q = wl.batch(w, 0, device="cuda")
    with new_cache(w, L.LACACHE_STAGE1_LSH) as cache:
        fill(cache, w)
        with pytest.raises(L.LacacheError) as e:
            cache.lookup(q["emb"], q["prefix"], q["ids"])
        assert e.value.status == L.LACACHE_ERR_INVALID_ARG
        L.lacache_enable_lsh(cache.h, 256, 256, wl.hyperplanes(256, w.d, device="cuda"))
        out = cache.lookup(q["emb"], q["prefix"], q["ids"])
        torch.cuda.synchronize()
        assert out["status"].shape == (w.batch,)
