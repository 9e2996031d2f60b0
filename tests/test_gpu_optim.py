"""GPU vs oracle: the update of the learnable factors that closes each calibration step
(App. B.1's AdamW with the linear learning-rate decay; §2.2's constraints as a projection),
through catq_factor_adamw_step.

Both sides take the same fp32 factors, gradients and hyperparameters; the oracle carries
its state in fp64 across updates.  Bar: fp32 max relative error per tensor.  The cases
cover one group, a ragged count that is no multiple of a block, the group count of the
Llama-3-8B-shaped gate_proj (14336 x 4096 / 128), factors pushed across every bound of the
projection, and a NaN gradient, which must surface as a NaN factor, not be clipped."""
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


def _f32(x):
    return float(np.float32(x))


@pytest.mark.parametrize("G,wd,margin,edges", [(1, 0.0, 1e-4, False), (1000, 0.0, 1e-4, True),
                                               (4099, 0.01, 1e-3, True), (458752, 0.0, 1e-4, False)])
def test_factor_adamw_step_matches_oracle(device, G, wd, margin, edges):
    import torch

    from paper_2606_26650_gb300 import catq as C
    tag = f"adamw/{G}"
    fac = [f.copy() for f in syn.factors(G, 0, tag, perturbed=True)]
    if edges and G >= 8:
        # near every bound, with gradients that push across it
        fac[0][:2] = [1 - 1.5 * margin, -1 + 1.5 * margin]
        fac[1][2:4] = 1.5 * margin
        fac[2][4:6] = 1.5 * margin
    hp = C.adamw(beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=wd, margin=margin)
    b1, b2, eps, wd32, m32 = (_f32(v) for v in (0.9, 0.999, 1e-8, wd, margin))
    dev_f = [torch.from_numpy(f).to(device) for f in fac]
    moments = torch.zeros(6 * G, dtype=torch.float32, device=device)
    ref_f = tuple(f.astype(np.float64) for f in fac)
    ref_m = (np.zeros(G),) * 6
    total = 5
    for k in range(total):
        grads = [g.copy() for g in syn.gradients(G, k, tag)]
        if edges and G >= 8:
            grads[0][:2] = [-1e-3, 1e-3]  # d_mu up past 1 - margin, down past -1 + margin
            grads[1][2:4] = 1e-3          # d_alpha, d_delta down past margin
            grads[2][4:6] = 1e-3
        lr = C.catq_linear_decay_lr(1e-3, k, total)
        dev_g = [torch.from_numpy(g).to(device) for g in grads]
        C.catq_factor_adamw_step(*dev_f, *dev_g, moments, hp, k + 1, lr)
        ref_f, ref_m = O.factor_update(ref_f, [g.astype(np.float64) for g in grads], ref_m, k + 1, _f32(lr),
                                       b1, b2, eps, wd32, m32)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    got_m = moments.cpu().numpy().reshape(6, G)
    errs = {}
    for q, name in enumerate(("d_mu", "d_alpha", "d_delta")):
        errs[name] = U.max_rel(dev_f[q].cpu().numpy(), ref_f[q])
        errs["m_" + name] = U.max_rel(got_m[q], ref_m[q])
        errs["v_" + name] = U.max_rel(got_m[3 + q], ref_m[3 + q])
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_F32}
    assert not bad, f"tolerance {U.TOL_F32} exceeded: {bad}"
    if edges and G >= 8:
        got = [f.cpu().numpy() for f in dev_f]
        np.testing.assert_allclose(got[0][:2], [1 - margin, -1 + margin], rtol=1e-7)
        np.testing.assert_allclose(got[1][2:4], margin, rtol=1e-7)
        np.testing.assert_allclose(got[2][4:6], margin, rtol=1e-7)
        assert all(np.isfinite(f).all() for f in got)
        assert np.all(got[0] >= np.float32(-1 + margin)) and np.all(got[0] <= np.float32(1 - margin))
        assert np.all(got[1] >= np.float32(margin)) and np.all(got[2] >= np.float32(margin))


def test_factor_adamw_step_nan_gradient_is_not_hidden(device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    G = 300
    fac = [torch.from_numpy(f.copy()).to(device) for f in syn.factors(G, 1, "adamw/nan", perturbed=True)]
    grads = [torch.from_numpy(g.copy()).to(device) for g in syn.gradients(G, 1, "adamw/nan")]
    grads[1][7] = float("nan")
    moments = torch.zeros(6 * G, dtype=torch.float32, device=device)
    C.catq_factor_adamw_step(*fac, *grads, moments, C.adamw(), 1, 1e-3)
    torch.cuda.synchronize()
    a = fac[1].cpu().numpy()
    assert np.isnan(a[7]) and np.isfinite(np.delete(a, 7)).all()
    assert np.isfinite(fac[0].cpu().numpy()).all() and np.isfinite(fac[2].cpu().numpy()).all()
