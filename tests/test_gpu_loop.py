"""GPU vs oracle parity of the composed calibration loop (App. B.1 with §2.3's schedule):
epochs of calibration steps, each the forward, the Eq. 7 loss, the backward and the AdamW
update of the three factors (catq_factor_adamw_step) at the linearly decayed learning rate,
with (phase, s) from catq_schedule_at_epoch, run on the GPU through the C ABI and in the
fp64 oracle from the same seeded inputs.

* fp32 (the oracle pin's own setting: 60 epochs x 3 batches of a 16 x 64 layer, g = 16):
  every per-step loss within max relative error 1e-5, and the factors after the loop within
  1e-5 of their size; the hard-ternarized loss after the loop below 0.9 of the start's on
  both sides.
* bf16 (256 x 512, g = 128, 3 batches of 100 tokens, 20 epochs): per-step losses within 2e-2,
  and the factors' total movement (end minus start) within 2e-2 relative Frobenius error,
  the bar of the gradients the loop integrates.
"""
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


def _oracle_loop(W, X, g, m, batches, gamma, s0, lr0):
    stats = O.group_stats(W, g)
    G = W.size // g
    fac, mom = (np.zeros(G), np.ones(G), np.ones(G)), (np.zeros(G),) * 6
    losses, t = [], 0
    for e in range(1, m + 1):
        phase, s = O.schedule_at_epoch(e, m, gamma, s0)
        for b in range(batches):
            step = O.calibration_step(X[b::batches], W, g, stats, fac, phase, s)
            losses.append(step["loss"])
            lr = O.linear_decay_lr(lr0, t, m * batches)
            t += 1
            fac, mom = O.factor_update(fac, (step["g_dmu"], step["g_dalpha"], step["g_ddelta"]), mom, t, lr)
    return stats, fac, np.array(losses)


def _gpu_loop(W, X, g, dtype, m, batches, gamma, s0, lr0, device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    N, K = W.shape
    G = N * K // g
    layer = C.Layer.create(U.to_device(W, dtype, device), g)
    C.catq_group_stats(layer)
    moments = torch.zeros(6 * G, dtype=torch.float32, device=device)
    hp = C.adamw()
    xs = [U.to_device(np.ascontiguousarray(X[b::batches]), dtype, device) for b in range(batches)]
    dt = layer.W.dtype
    yts = []
    for xb in xs:
        yt = torch.empty(xb.shape[0], N, dtype=dt, device=device)
        C.catq_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), xb, yt)
        yts.append(yt)
    grads = [torch.empty(G, dtype=torch.float32, device=device) for _ in range(3)]
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    losses = torch.zeros(m * batches, dtype=torch.float32, device=device)
    t = 0
    for e in range(1, m + 1):
        sched = C.catq_schedule_at_epoch(e, m, gamma, s0)
        for b, (xb, yt) in enumerate(zip(xs, yts)):
            Y = torch.empty_like(yt)
            dY = torch.empty_like(yt)
            C.catq_soft_ternary_linear_fwd(layer, sched, xb, Y)
            C.catq_recon_loss(Y, yt, loss, dY, C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), device))
            losses[t].copy_(loss[0])
            C.catq_soft_ternary_linear_bwd(layer, sched, xb, dY, None, *grads,
                                           workspace=C.workspace(C.catq_bwd_workspace_bytes(layer, xb.shape[0]),
                                                                 device))
            lr = C.catq_linear_decay_lr(lr0, t, m * batches)
            t += 1
            C.catq_factor_adamw_step(layer.d_mu, layer.d_alpha, layer.d_delta, *grads, moments, hp, t, lr)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    fac = tuple(U.to_host(f).astype(np.float64) for f in (layer.d_mu, layer.d_alpha, layer.d_delta))
    return fac, U.to_host(losses).astype(np.float64)


def test_loop_fp32_at_the_oracle_pins_setting(device):
    r = np.random.default_rng(0)
    N, K, g, M = 16, 64, 16, 96
    W = r.standard_normal((N, K)) * 0.02
    X = r.standard_normal((M, K))
    W32, X32 = W.astype(np.float32), X.astype(np.float32)
    m, batches = 60, 3
    stats, fac_o, loss_o = _oracle_loop(W32.astype(np.float64), X32.astype(np.float64), g, m, batches, 0.8, 30.0,
                                        1e-3)
    fac_g, loss_g = _gpu_loop(W32, X32, g, "f32", m, batches, 0.8, 30.0, 1e-3, device)
    rel = np.abs(loss_g - loss_o) / np.abs(loss_o)
    assert rel.max() <= 1e-5, rel.max()
    for name, a, b in zip(("d_mu", "d_alpha", "d_delta"), fac_g, fac_o):
        err = np.abs(a - b).max() / np.abs(b).max()
        assert err <= 1e-5, (name, err)

    def hard_loss(f):
        return O.calibration_step(X32.astype(np.float64), W32.astype(np.float64), g, stats, f, O.PHASE_HARD,
                                  30.0)["loss"]

    start = hard_loss((np.zeros(W.size // g), np.ones(W.size // g), np.ones(W.size // g)))
    assert hard_loss(fac_g) < 0.9 * start and hard_loss(fac_o) < 0.9 * start


def test_loop_bf16(device):
    r = syn.rng(60, "loop/bf16")
    N, K, g, batches = 256, 512, 128, 3
    M = 100 * batches
    W = syn.round_bf16((r.standard_normal((N, K)) * 0.02).astype(np.float32))
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    m = 20
    _, fac_o, loss_o = _oracle_loop(W.astype(np.float64), X.astype(np.float64), g, m, batches, 0.8, 30.0, 1e-3)
    fac_g, loss_g = _gpu_loop(W, X, g, "bf16", m, batches, 0.8, 30.0, 1e-3, device)
    rel = np.abs(loss_g - loss_o) / np.abs(loss_o)
    G = N * K // g
    start = (np.zeros(G), np.ones(G), np.ones(G))
    moves = {name: U.fro_rel(a - s, b - s) for name, a, b, s in zip(("d_mu", "d_alpha", "d_delta"), fac_g, fac_o,
                                                                       start)}
    print(f"bf16 loop: worst step loss error {rel.max():.3e}, factor movement errors {moves}, "
          f"loss {loss_o[0]:.4e} -> {loss_o[-1]:.4e}")
    assert rel.max() <= U.TOL_BF16, rel.max()
    bad = {k: v for k, v in moves.items() if not v <= U.TOL_BF16}
    assert not bad, moves
