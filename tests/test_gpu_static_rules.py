"""GPU parity of §2.2's static scale/threshold rules (absmean, TWN) used as base statistics:
the statistics themselves, then a whole SOFT calibration step from them.  For TWN the GPU
compares |W_i| with 0.7 mean|W| in fp32 and the oracle in fp64, so a group holding an
element within 1e-5 (relative) of that threshold may count it on the other side; such
groups are left out of the statistics comparison (as near-threshold codes are elsewhere)."""
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


def _near_twn_threshold(W, g):
    Wg = np.abs(W.astype(np.float64)).reshape(-1, g)
    dW = 0.7 * Wg.mean(axis=1)
    return (np.abs(Wg - dW[:, None]) <= 1e-5 * dW[:, None]).any(axis=1)


@pytest.mark.parametrize("rule", [O.THR_ABSMEAN, O.THR_TWN_STATIC])
@pytest.mark.parametrize("N,K,g,M", [(1024, 4096, 128, 1100),   # register (team) kernel, four-CTA GEMMs
                                     (64, 4096, 4096, 300)])     # channel-wise: streaming kernel
def test_static_rule_stats_and_step(device, rule, N, K, g, M):
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = syn.WORKLOADS["c3_llama3_8b_block"]
    r = syn.rng(9, f"static/{rule}/{N}/{K}/{g}")
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * wl.w_std)
    X = syn.activations(wl, "x_hidden", M, K)
    G = N * K // g
    fac = syn.factors(G, 9, f"static/{N}/{K}", perturbed=True)

    layer = C.Layer.create(U.to_device(W, "bf16", device), g)
    C.catq_group_stats(layer, rule)
    torch.cuda.synchronize()
    want = O.group_stats(W, g, rule)
    keep = ~_near_twn_threshold(W, g) if rule == O.THR_TWN_STATIC else np.ones(G, bool)
    assert keep.mean() > 0.99
    np.testing.assert_array_equal(U.to_host(layer.mu0), 0.0)
    np.testing.assert_allclose(U.to_host(layer.alpha0)[keep], want[1][keep], rtol=1e-6)
    np.testing.assert_allclose(U.to_host(layer.delta0)[keep], want[2][keep], rtol=1e-6)

    got = U.gpu_step(W, X, g, fac, rule, O.PHASE_SOFT, 30.0, "bf16", device)
    ref = O.calibration_step(X, W, g, want, fac, O.PHASE_SOFT, 30.0)
    errs = {k: U.fro_rel(got[k], ref[k]) for k in ("Y", "dY", "dX", "g_dmu", "g_dalpha", "g_ddelta")}
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, f"tolerance {U.TOL_BF16} exceeded: {bad} (all: {errs})"
