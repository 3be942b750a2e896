"""GPU parity of threshold calibration (App. A.2) against the oracle: pair similarities within 2e-3, and the
nearest-rank percentile and capped threshold of the GPU's similarities against the oracle's."""
import numpy as np
import pytest
import torch

import oracle
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


def _gpu(x, y, percentile, cap):
    sims = torch.empty(x.shape[0], dtype=torch.float32, device="cuda")
    res = torch.empty(2, dtype=torch.float32, device="cuda")
    ws = torch.empty(L.lacache_calibrate_workspace_bytes(), dtype=torch.uint8, device="cuda")
    L.lacache_calibrate(x, y, percentile, cap, sims, res, ws)
    torch.cuda.synchronize()
    return sims.cpu().numpy(), res.cpu().numpy()


def test_exact_dyadic_pairs_are_bit_exact():
    e = np.eye(8)
    base = [e[0], e[0], e[1], np.r_[[0.5] * 4, [0] * 4], e[2]]
    other = [e[0], np.r_[0.75, 0.5, 0.25, [0] * 5], e[3], np.r_[[0.5] * 4, [0] * 4], -e[2]]
    x = torch.tensor(np.array(base), dtype=torch.bfloat16, device="cuda")
    y = torch.tensor(np.array(other), dtype=torch.bfloat16, device="cuda")
    ox, oy = oracle.round_to_bf16(np.array(base, np.float32)), oracle.round_to_bf16(np.array(other, np.float32))
    for pct, cap in [(0, 0.8), (20, 0.8), (50, 0.8), (60, 0.5), (100, 0.8), (100, 2.0)]:
        sims, res = _gpu(x, y, pct, cap)
        tau, p = oracle.calibrate(ox, oy, pct, float(np.float32(cap)))     # the cap is passed as a float32
        assert list(sims) == list(oracle.pair_similarities(ox, oy))
        assert (float(res[0]), float(res[1])) == (p, tau), pct


@pytest.mark.parametrize("n", [1, 500, 200_000])
@pytest.mark.parametrize("pct,cap", [(5, 0.80), (10, 0.70), (10, 0.99)])
def test_benign_pairs_match_the_oracle(n, pct, cap):
    x, y = wl.benign_pairs(n, 1024, 0.6, device="cuda")
    sims, res = _gpu(x, y, pct, cap)
    ox, oy = wl.bf16_bits(x), wl.bf16_bits(y)
    osims = oracle.pair_similarities(ox, oy)
    assert np.max(np.abs(sims - osims)) <= TOL
    tau, p = oracle.calibrate(ox, oy, pct, float(np.float32(cap)))
    assert abs(res[0] - p) <= TOL and abs(res[1] - tau) <= TOL
    # the GPU's value is exactly the nearest-rank percentile of the GPU's own similarities
    assert res[0] == oracle.nearest_rank(sims.astype(np.float64), pct)


def test_ties_and_invalid_arguments():
    x = torch.tensor(np.eye(8)[[0] * 64], dtype=torch.bfloat16, device="cuda")
    sims, res = _gpu(x, x, 37.5, 0.9)
    assert np.all(sims == 1.0) and list(res) == [1.0, pytest.approx(0.9)]
    with pytest.raises(L.LacacheError) as e:
        _gpu(x, x, 101, 0.9)
    assert e.value.status == L.LACACHE_ERR_INVALID_ARG
