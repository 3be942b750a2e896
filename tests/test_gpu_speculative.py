"""GPU parity of the draft-verification bookkeeping (section 3.3) against the oracle: accepted prefix lengths
are integers decided by fp32 comparisons of the same fp32 inputs on both sides, so they must agree exactly."""
import numpy as np
import pytest
import torch

import oracle
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


@pytest.mark.parametrize("B,k", [(1, 1), (37, 20), (256, 32), (1000, 33), (64, 256)])
def test_accepted_prefix_matches_the_oracle(B, k):
    pf, pg = wl.draft_probabilities(B, k, device="cuda")
    status = torch.randint(0, 3, (B,), dtype=torch.uint8, device="cuda")
    acc = torch.empty(B, dtype=torch.int32, device="cuda")
    L.lacache_verify_draft(pf, pg, status, acc)
    acc_all = torch.empty(B, dtype=torch.int32, device="cuda")
    L.lacache_verify_draft(pf, pg, None, acc_all)
    torch.cuda.synchronize()
    hpf, hpg = pf.cpu().numpy(), pg.cpu().numpy()
    assert np.array_equal(acc.cpu().numpy(), oracle.accepted_prefix(hpf, hpg, status.cpu().numpy()))
    want = oracle.accepted_prefix(hpf, hpg)
    assert np.array_equal(acc_all.cpu().numpy(), want)
    if B >= 256 and k <= 64:
        assert want.min() == 0 and want.max() == k        # rejections at the first token and full acceptances
