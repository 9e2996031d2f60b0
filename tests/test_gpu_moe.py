"""Config 5 (MoE layer) parity: every expert's soft-ternary forward/backward through the
grouped C calls against the oracle, per expert, on expert-sorted rows.

The layer keeps the per-expert shapes (gate/up 4096 -> 1536, down 1536 -> 4096) and the
Zipf(1.1) Gumbel-top-k routing, with fewer experts and tokens than the full layer so the
fp64 oracle stays within seconds; the routing is skewed enough that some experts get many
rows, some a few and some none.
"""
import dataclasses

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


def _workload():
    base = syn.WORKLOADS["c5_qwen3_235b_moe"]
    return dataclasses.replace(base, experts=24, top_k=2, tokens=96)


@pytest.mark.parametrize("lin_name", ["gate_proj", "down_proj"])
@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 30.0), (O.PHASE_HARD, 30.0)])
def test_moe_grouped_matches_oracle(device, lin_name, phase, s):
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = _workload()
    lin = wl.linear(lin_name)
    E, N, K, g = wl.experts, lin.N, lin.K, wl.g
    token_of_row, off = syn.moe_routing(wl, seed=0)
    R = int(off[-1])
    counts = np.diff(off)
    assert counts.max() > 3 * max(1, int(np.median(counts)))  # skewed routing
    W = np.stack([syn.weight(wl, lin, expert=e) for e in range(E)])
    X_tok = syn.activations(wl, lin.x, wl.tokens, K)
    X = X_tok[token_of_row]
    G = N * K // g
    fac = syn.factors(E * G, 0, f"moe/{lin_name}", perturbed=True)

    Wt = U.to_device(W.reshape(E * N, K), "bf16", device).reshape(E, N, K)
    layer = C.GroupedLayer.create(Wt, g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer.dense)
    Xt = U.to_device(X, "bf16", device)
    Yt = torch.empty(R, N, dtype=torch.bfloat16, device=device)
    Y = torch.empty_like(Yt)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), Xt, off, Yt)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(phase, s), Xt, off, Y)
    loss = torch.zeros(1, device=device)
    dY = torch.empty_like(Y)
    C.catq_recon_loss(Y, Yt, loss, dY, C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), device))
    dX = torch.empty_like(Xt)
    gr = [torch.empty(E * G, device=device) for _ in range(3)]
    ws = C.workspace(C.catq_grouped_bwd_workspace_bytes(layer, off), device)
    C.catq_grouped_soft_ternary_linear_bwd(layer, C.schedule(phase, s), Xt, dY, off, dX, *gr, ws)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0

    # oracle, expert by expert, with the loss normalised over all R x N outputs
    Y_ref = np.zeros((R, N))
    dX_ref = np.zeros((R, K))
    g_ref = [np.zeros(E * G) for _ in range(3)]
    Y_all, Yt_all = [], []
    stats_all = []
    for e in range(E):
        st = O.group_stats(W[e], g, O.THR_HALF)
        fe = tuple(f[e * G:(e + 1) * G] for f in fac)
        rows = slice(off[e], off[e + 1])
        Wq = O.ternary_weight(W[e], g, st, fe, phase, s)[0]
        Y_ref[rows] = O.linear_fwd(X[rows], Wq)
        Y_all.append(Y_ref[rows])
        Yt_all.append(O.linear_fwd(X[rows], W[e]))
        stats_all.append((st, fe))
    Yt_ref = np.concatenate(Yt_all) if R else np.zeros((0, N))
    loss_ref, dY_ref = O.recon_loss(Y_ref, Yt_ref)
    for e in range(E):
        st, fe = stats_all[e]
        rows = slice(off[e], off[e + 1])
        dxe, gm, ga, gd = O.linear_bwd(X[rows], dY_ref[rows], W[e], g, st, fe, phase, s)
        dX_ref[rows] = dxe
        for dst, src in zip(g_ref, (gm, ga, gd)):
            dst[e * G:(e + 1) * G] = src
    errs = {"Y": U.fro_rel(U.to_host(Y), Y_ref), "dX": U.fro_rel(U.to_host(dX), dX_ref),
            "loss": abs(loss.item() - loss_ref) / loss_ref}
    for name, got, ref in zip(("g_dmu", "g_dalpha", "g_ddelta"), gr, g_ref):
        errs[name] = U.fro_rel(U.to_host(got), ref)
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, errs
    empty = np.nonzero(counts == 0)[0]
    for e in empty:
        assert not U.to_host(gr[0])[e * G:(e + 1) * G].any()


@pytest.mark.parametrize("E", [128, 130])
def test_many_small_experts(device, E):
    """Many experts with a handful of rows each (some none): 128 experts run as grouped
    launches (dW in two launches of 64), 130 take the expert-by-expert path; both against
    the oracle."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    N, K, g = 256, 512, 128
    r = syn.rng(11, f"moe/many/{E}")
    counts = r.integers(0, 9, size=E)
    counts[::7] = 0
    off = np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)
    R = int(off[-1])
    W = syn.round_bf16((r.standard_normal((E, N, K)) * 0.02).astype(np.float32))
    X = syn.round_bf16(r.standard_normal((R, K)).astype(np.float32))
    dY = syn.round_bf16((r.standard_normal((R, N)) * 1e-2).astype(np.float32))
    G = N * K // g
    fac = syn.factors(E * G, 11, f"moe/many/{E}", perturbed=True)
    phase, s = O.PHASE_SOFT, 30.0
    Wt = U.to_device(W.reshape(E * N, K), "bf16", device).reshape(E, N, K)
    layer = C.GroupedLayer.create(Wt, g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer.dense)
    Xt, dYt = U.to_device(X, "bf16", device), U.to_device(dY, "bf16", device)
    Y = torch.empty(R, N, dtype=torch.bfloat16, device=device)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(phase, s), Xt, off, Y)
    dX = torch.empty_like(Xt)
    gr = [torch.full((E * G,), 7.0, device=device) for _ in range(3)]
    ws = C.workspace(C.catq_grouped_bwd_workspace_bytes(layer, off), device)
    C.catq_grouped_soft_ternary_linear_bwd(layer, C.schedule(phase, s), Xt, dYt, off, dX, *gr, ws)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    Yh, dXh = U.to_host(Y), U.to_host(dX)
    grh = [U.to_host(t) for t in gr]
    Y_ref, dX_ref = np.zeros((R, N)), np.zeros((R, K))
    g_ref = [np.zeros(E * G) for _ in range(3)]
    for e in range(E):
        rows = slice(int(off[e]), int(off[e + 1]))
        st = O.group_stats(W[e], g)
        fe = tuple(f[e * G:(e + 1) * G] for f in fac)
        Wq = O.ternary_weight(W[e], g, st, fe, phase, s)[0]
        Y_ref[rows] = O.linear_fwd(X[rows], Wq)
        dxe, *ge = O.linear_bwd(X[rows], dY[rows], W[e], g, st, fe, phase, s)
        dX_ref[rows] = dxe
        for dst, src in zip(g_ref, ge):
            dst[e * G:(e + 1) * G] = src
    errs = {"Y": U.fro_rel(Yh, Y_ref), "dX": U.fro_rel(dXh, dX_ref)}
    for name, got, want in zip(("g_dmu", "g_dalpha", "g_ddelta"), grh, g_ref):
        errs[name] = U.fro_rel(got, want)
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, errs
    for e in np.nonzero(counts == 0)[0]:
        assert not grh[0][e * G:(e + 1) * G].any() and not grh[2][e * G:(e + 1) * G].any()
