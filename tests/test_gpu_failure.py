"""Device-side failure detection on the GPU, without a fault: a bounded wait that nothing
satisfies gives up after its limit, latches CATQ_ERR_TIMEOUT, and leaves the context usable."""
import numpy as np
import pytest

from oracle import catq_oracle as O
from paper_2606_26650_gb300 import synthetic as syn
from tests import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def device():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.device("cuda:0")


def test_expired_wait_is_reported_and_the_context_survives(device):
    import time

    from paper_2606_26650_gb300 import catq as C
    assert C.catq_device_status() == 0
    t0 = time.perf_counter()
    C.catq_selftest_wait_timeout(5_000_000)  # 5 ms
    status = C.catq_device_status()  # synchronises
    elapsed = time.perf_counter() - t0
    assert C.STATUS[status] == "CATQ_ERR_TIMEOUT"
    assert elapsed >= 0.005
    assert C.catq_device_status() == 0  # reading cleared it

    # the next calls run normally and stay correct
    r = syn.rng(3, "after-timeout")
    N, K, g, M = 256, 512, 128, 1100
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 3, "after-timeout", perturbed=True)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16", device)
    stats = O.group_stats(W, g, O.THR_HALF)
    ref = O.calibration_step(X, W, g, stats, fac, O.PHASE_SOFT, 30.0)
    for k in ("Y", "dX", "g_dmu"):
        assert U.fro_rel(got[k], ref[k]) <= U.TOL_BF16, k
