"""Helpers shared by the GPU parity tests: device upload of the seeded inputs, the
error measures of the acceptance bar, and one full calibration step through the C ABI."""
from __future__ import annotations

import numpy as np

from paper_2606_26650_gb300 import synthetic as syn

# Acceptance bar: fp32 max relative error (max |a-b| / max |b| per tensor); bf16 relative
# Frobenius error; ternary codes bit-exact outside the 1e-6 relative threshold band.
TOL_F32 = 1e-5
TOL_BF16 = 2e-2
NEAR_THRESHOLD = 1e-6


def max_rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    den = np.abs(b).max()
    return float(np.abs(a - b).max() / (den if den > 0 else 1.0))


def fro_rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    den = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (den if den > 0 else 1.0))


def err(a, b, dtype: str) -> float:
    return max_rel(a, b) if dtype == "f32" else fro_rel(a, b)


def tol(dtype: str) -> float:
    return TOL_F32 if dtype == "f32" else TOL_BF16


def to_device(a: np.ndarray, dtype: str, device):
    import torch
    if dtype == "bf16":
        return torch.from_numpy(syn.bf16_bits(a).view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)


def to_host(t) -> np.ndarray:
    import torch
    if t.dtype == torch.bfloat16:
        return t.float().cpu().numpy()
    return t.cpu().numpy()


def gpu_step(W, X, g, fac, thr, phase, s, dtype, device, with_dx=True, recon=0):
    """Group stats, teacher and phase forward, loss, backward and hard pack on the GPU
    (`recon` 1: the W ~ alpha T + mu reconstruction).  Returns a dict of host arrays."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    M, K = X.shape
    N = W.shape[0]
    G = N * K // g
    Wt, Xt = to_device(W, dtype, device), to_device(X, dtype, device)
    layer = C.Layer.create(Wt, g, *(torch.from_numpy(np.asarray(f, np.float32)).to(device) for f in fac),
                           recon=recon)
    C.catq_group_stats(layer, thr)
    tdt = Wt.dtype
    Yref = torch.empty(M, N, dtype=tdt, device=device)
    Y = torch.empty_like(Yref)
    C.catq_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), Xt, Yref)
    C.catq_soft_ternary_linear_fwd(layer, C.schedule(phase, s), Xt, Y)
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    dY = torch.empty_like(Y)
    ws = C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), device)
    C.catq_recon_loss(Y, Yref, loss, dY, ws)
    dX = torch.empty_like(Xt) if with_dx else None
    gr = [torch.empty(G, dtype=torch.float32, device=device) for _ in range(3)]
    wsb = C.workspace(C.catq_bwd_workspace_bytes(layer, M), device)
    C.catq_soft_ternary_linear_bwd(layer, C.schedule(phase, s), Xt, dY, dX, *gr, wsb)
    codes = torch.empty(N * K // 4, dtype=torch.uint8, device=device)
    alpha = torch.empty(G, dtype=torch.float32, device=device)
    mu = torch.empty(G, dtype=torch.float32, device=device)
    C.catq_hard_ternarize_pack(layer, codes, alpha, mu)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    out = dict(mu0=to_host(layer.mu0), alpha0=to_host(layer.alpha0), delta0=to_host(layer.delta0),
               Y_ref=to_host(Yref), Y=to_host(Y), loss=float(loss.item()), dY=to_host(dY),
               g_dmu=to_host(gr[0]), g_dalpha=to_host(gr[1]), g_ddelta=to_host(gr[2]),
               codes=to_host(codes), alpha=to_host(alpha), mu=to_host(mu))
    if with_dx:
        out["dX"] = to_host(dX)
    return out
