"""GPU vs oracle for direct learning (DL) and the synthetic analogue of Fig. fig:error (§2.2):
the DL update (catq_direct_adamw_step) against the oracle's ``direct_update`` over several
updates (fp32 max relative error 1e-5 per tensor), the per-group weight reconstruction error
(catq_group_recon_error) against ``group_recon_error`` on bf16 and fp32 layers, and the
three strategies of the figure run as calibration loops on the GPU and in the oracle from the
same seeded fp32 layer: the static absmean rule (SA), direct learning started from it (DL),
and the learnable modulation (LM), all with hard ternarization throughout as in the figure.
Their per-group errors must agree within 1e-4 of the largest, except in groups where a weight
reached its threshold within fp32 resolution during the loop: with hard ternarization that
weight's code is decided by the precision of the comparison (as in the 1e-6 band the code
comparisons excuse), and its group then follows another trajectory.  Such groups are counted,
listed with the other near-threshold listings and bounded (at most 2% of the groups), and
the mean and median error over all groups must still agree within 1e-4.  The test prints the
statistics of the three strategies."""
import os

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


@pytest.mark.parametrize("G,wd,margin", [(1, 0.0, 1e-4), (4099, 0.01, 1e-3), (32768, 0.0, 1e-4)])
def test_direct_update_matches_oracle(device, G, wd, margin):
    import torch

    from paper_2606_26650_gb300 import catq as C
    tag = f"direct/{G}"
    fac = [f.copy() for f in syn.factors(G, 0, tag, perturbed=True)]
    if G >= 8:
        fac[1][:2] = 1.5 * margin  # a pushed below its bound
    hp = C.adamw(beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=wd, margin=margin)
    dal = torch.from_numpy(fac[1]).to(device)
    ddl = torch.from_numpy(fac[2]).to(device)
    moments = torch.zeros(4 * G, dtype=torch.float32, device=device)
    ref_a, ref_d = fac[1].astype(np.float64), fac[2].astype(np.float64)
    ref_m = (np.zeros(G),) * 4
    total = 5
    for k in range(total):
        grads = [g.copy() for g in syn.gradients(G, k, tag)]
        if G >= 8:
            grads[1][:2] = 1e-3
        lr = C.catq_linear_decay_lr(1e-3, k, total)
        ga, gd = (torch.from_numpy(g).to(device) for g in grads[1:])
        C.catq_direct_adamw_step(dal, ddl, ga, gd, moments, hp, k + 1, lr)
        # the oracle carries its own fp64 state; the hyperparameters are the fp32 values the GPU uses
        ref_a, ref_d, ref_m = O.direct_update(ref_a, ref_d, grads[1].astype(np.float64), grads[2].astype(np.float64),
                                              ref_m, k + 1, _f32(lr), _f32(0.9), _f32(0.999), _f32(1e-8), _f32(wd),
                                              _f32(margin))
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    got_m = moments.cpu().numpy().reshape(4, G)
    errs = {"d_alpha": U.max_rel(dal.cpu().numpy(), ref_a), "d_delta": U.max_rel(ddl.cpu().numpy(), ref_d)}
    for q, name in enumerate(("m_a", "m_d", "v_a", "v_d")):
        errs[name] = U.max_rel(got_m[q], ref_m[q])
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_F32}
    assert not bad, f"tolerance {U.TOL_F32} exceeded: {bad}"
    if G >= 8:
        assert np.all(dal.cpu().numpy() >= np.float32(margin))


@pytest.mark.parametrize("dtype,N,K,g,thr", [("bf16", 1024, 4096, 128, O.THR_ABSMEAN), ("bf16", 328, 384, 128, O.THR_HALF),
                                             ("f32", 64, 96, 32, O.THR_TWN07)])
def test_group_recon_error_matches_oracle(device, dtype, N, K, g, thr):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(72, f"recon_err/{dtype}/{N}")
    W = (r.standard_normal((N, K)) * 0.02).astype(np.float32)
    if dtype == "bf16":
        W = syn.round_bf16(W)
    G = N * K // g
    fac = syn.factors(G, 72, f"recon_err/{N}", perturbed=True)
    layer = C.Layer.create(U.to_device(W, dtype, device), g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer, thr)
    err = torch.empty(G, dtype=torch.float32, device=device)
    C.catq_group_recon_error(layer, err)
    torch.cuda.synchronize()
    stats = O.group_stats(W, g, thr)
    want = O.group_recon_error(W, g, stats, fac)
    _, _, gap = O.hard_codes(W, g, stats, fac)
    clean = ~(gap.reshape(G, g) <= U.NEAR_THRESHOLD).any(axis=1)  # no code within the threshold band
    got = U.to_host(err)
    assert U.max_rel(got[clean], want[clean]) <= U.TOL_F32


def _oracle_strategy(kind, W, X, g, m, batches, lr0, s0):
    """SA: the absmean rule as is.  DL: started from it, DL's own AdamW.  LM: Eq. 3's
    statistics and the modulation's AdamW.  Hard ternarization throughout."""
    G = W.size // g
    stats = O.group_stats(W, g, O.THR_HALF if kind == "LM" else O.THR_ABSMEAN)
    fac = (np.zeros(G), np.ones(G), np.ones(G))
    if kind != "SA":
        mom = (np.zeros(G),) * (6 if kind == "LM" else 4)
        t = 0
        for _ in range(m):
            for b in range(batches):
                step = O.calibration_step(X[b::batches], W, g, stats, fac, O.PHASE_HARD, s0)
                lr = O.linear_decay_lr(lr0, t, m * batches)
                t += 1
                if kind == "LM":
                    fac, mom = O.factor_update(fac, (step["g_dmu"], step["g_dalpha"], step["g_ddelta"]), mom, t, lr)
                else:
                    a, d, mom = O.direct_update(fac[1], fac[2], step["g_dalpha"], step["g_ddelta"], mom, t, lr)
                    fac = (fac[0], a, d)
    return O.group_recon_error(W, g, stats, fac)


def _gpu_strategy(kind, W, X, g, m, batches, lr0, s0, device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    N, K = W.shape
    G = N * K // g
    layer = C.Layer.create(U.to_device(W, "f32", device), g)
    C.catq_group_stats(layer, C.THR_HALF if kind == "LM" else C.THR_ABSMEAN)
    if kind != "SA":
        hp = C.adamw()
        moments = torch.zeros((6 if kind == "LM" else 4) * G, dtype=torch.float32, device=device)
        xs = [U.to_device(np.ascontiguousarray(X[b::batches]), "f32", device) for b in range(batches)]
        yts = []
        for xb in xs:
            yt = torch.empty(xb.shape[0], N, dtype=torch.float32, device=device)
            C.catq_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), xb, yt)
            yts.append(yt)
        grads = [torch.empty(G, dtype=torch.float32, device=device) for _ in range(3)]
        loss = torch.zeros(1, dtype=torch.float32, device=device)
        sched = C.schedule(C.PHASE_HARD, s0)
        t = 0
        for _ in range(m):
            for xb, yt in zip(xs, yts):
                Y, dY = torch.empty_like(yt), torch.empty_like(yt)
                C.catq_soft_ternary_linear_fwd(layer, sched, xb, Y)
                C.catq_recon_loss(Y, yt, loss, dY, C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), device))
                C.catq_soft_ternary_linear_bwd(layer, sched, xb, dY, None, *grads,
                                               workspace=C.workspace(C.catq_bwd_workspace_bytes(layer, xb.shape[0]),
                                                                     device))
                lr = C.catq_linear_decay_lr(lr0, t, m * batches)
                t += 1
                if kind == "LM":
                    C.catq_factor_adamw_step(layer.d_mu, layer.d_alpha, layer.d_delta, *grads, moments, hp, t, lr)
                else:
                    C.catq_direct_adamw_step(layer.d_alpha, layer.d_delta, grads[1], grads[2], moments, hp, t, lr)
    err = torch.empty(G, dtype=torch.float32, device=device)
    C.catq_group_recon_error(layer, err)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    return U.to_host(err).astype(np.float64)


def test_fig_error_strategies_fp32(device):
    r = syn.rng(73, "fig_error")
    N, K, g, batches = 64, 256, 64, 3
    W = (r.standard_normal((N, K)) * 0.02).astype(np.float32)
    X = r.standard_normal((96 * batches, K)).astype(np.float32)
    m, lr0, s0 = 20, 1e-3, 30.0
    stats = {}
    for kind in ("SA", "DL", "LM"):
        want = _oracle_strategy(kind, W.astype(np.float64), X.astype(np.float64), g, m, batches, lr0, s0)
        got = _gpu_strategy(kind, W, X, g, m, batches, lr0, s0, device)
        rel = np.abs(got - want) / np.abs(want).max()
        diverged = np.nonzero(rel > 1e-4)[0]
        with open(os.path.join(U.listing_dir(), f"fig_error_{kind}_diverged_groups.txt"), "w") as fh:
            fh.write(f"# {kind}: {diverged.size} of {rel.size} groups whose error differs by more than 1e-4\n")
            for j in diverged:
                fh.write(f"{j} {want[j]:.6e} {got[j]:.6e}\n")
        assert diverged.size <= max(1, rel.size // 50), (kind, diverged.size)
        assert abs(got.mean() - want.mean()) <= 1e-4 * want.mean(), kind
        assert abs(np.median(got) - np.median(want)) <= 1e-4 * np.median(want), kind
        stats[kind] = (float(np.mean(got)), float(np.median(got)), float(np.max(got)), int(diverged.size))
    print("per-group weight reconstruction error (mean, median, max, diverged groups):", stats)
    # calibration moves both learned strategies away from the static rule
    assert stats["DL"][0] != stats["SA"][0] and stats["LM"][0] != stats["SA"][0]
