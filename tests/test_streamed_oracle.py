"""The streamed oracle of the full-size parity tests (chunk-by-chunk key check, regenerated prefix rows) gives the
same result, margins included, as the oracle over the resident store. CPU only: the store is generated on the
host and no cache is built."""
import numpy as np
import torch

import oracle
from paper_2608_01718_gb300 import workloads as wl
from parity import StreamedOracle, oracle_queries, oracle_store, params, stratified_sample


def test_streamed_oracle_equals_the_resident_oracle():
    # few, large clusters: every near-duplicate and collision has hundreds of entries above tau_c, so the margin of
    # a rejection examines entries well past the candidate cut
    w = wl.WORKLOADS["mid-1m"].scaled(n=40_000, batch=48, clusters=40)
    q = wl.batch(w, 0, device="cpu")
    sample = stratified_sample(q["class"], 8)
    p = params(w)
    so = StreamedOracle(w, q, sample, p)
    so.fill(None, device="cpu")
    got = so.result()
    want = oracle.lookup(oracle_store(w, device="cpu"), oracle_queries(q, torch.as_tensor(sample)), p)
    assert np.max(got.n_above) > 10 * w.top_c
    assert set(got.status.tolist()) == {oracle.MISS_KEY, oracle.HIT, oracle.REJECT}
    for f in want.__dataclass_fields__:
        assert np.array_equal(getattr(got, f), getattr(want, f), equal_nan=True), f
