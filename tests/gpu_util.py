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


def gpu_step(W, X, g, fac, thr, phase, s, dtype, device, with_dx=True, recon=0, fused=False, teacher_f32=False,
             a8=False, reduction=0):
    """Group stats, teacher and phase forward, loss, backward and hard pack on the GPU
    (`recon` 1: the W ~ alpha T + mu reconstruction).  `fused`: forward, loss and dY in one
    call (catq_soft_ternary_linear_fwd_loss); `teacher_f32`: the teacher output of a bf16
    layer kept in fp32 (fused only); `a8`: the layer's input quantized to 8 bits per token
    (codes and scales into the forward, the dequantized activations into dW; the teacher
    from the full-precision input).  Returns a dict of host arrays."""
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
    Xf, Xw, rs = Xt, Xt, None  # forward input, dW input, per-row scale
    extra = {}
    if a8:
        Xf, Xw = torch.empty_like(Xt), torch.empty_like(Xt)
        rs = torch.empty(M, dtype=torch.float32, device=device)
        C.catq_act_quant_a8(Xt, Xf, rs, Xw)
        extra = dict(a8_codes=Xf, a8_scale=rs, a8_deq=Xw)
    Yref = torch.empty(M, N, dtype=torch.float32 if teacher_f32 else tdt, device=device)
    Y = torch.empty(M, N, dtype=tdt, device=device)
    if teacher_f32:
        C.catq_soft_ternary_linear_fwd_ex(layer, C.schedule(C.PHASE_TEACHER), Xt, Yref)
    else:
        C.catq_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), Xt, Yref)
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    dY = torch.empty_like(Y)
    if fused:
        ws = C.workspace(C.catq_fwd_loss_workspace_bytes(layer, M), device)
        C.catq_soft_ternary_linear_fwd_loss(layer, C.schedule(phase, s), Xf, Yref, loss, dY, Y=Y, x_row_scale=rs,
                                            workspace=ws, reduction=reduction)
    else:
        assert not teacher_f32
        if rs is not None:
            C.catq_soft_ternary_linear_fwd_ex(layer, C.schedule(phase, s), Xf, Y, x_row_scale=rs)
        else:
            C.catq_soft_ternary_linear_fwd(layer, C.schedule(phase, s), Xf, Y)
        ws = C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), device)
        C.catq_recon_loss(Y, Yref, loss, dY, ws, reduction=reduction)
    dX = torch.empty_like(Xt) if with_dx else None
    gr = [torch.empty(G, dtype=torch.float32, device=device) for _ in range(3)]
    wsb = C.workspace(C.catq_bwd_workspace_bytes(layer, M), device)
    C.catq_soft_ternary_linear_bwd(layer, C.schedule(phase, s), Xw, dY, dX, *gr, wsb)
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
    for k, v in extra.items():
        out[k] = to_host(v)
    return out


def listing_dir():
    """Where the near-threshold listings go: $CATQ_LISTING_DIR, else catq_near_threshold/ under
    the system's temporary directory (never inside the repository)."""
    import os
    import tempfile
    d = os.environ.get("CATQ_LISTING_DIR") or os.path.join(tempfile.gettempdir(), "catq_near_threshold")
    os.makedirs(d, exist_ok=True)
    return d


def check_codes(got, want, gap, name=None, bound_frac=1e-5, bound_min=16):
    """Ternary codes are bit-exact except elements whose |What| lies within 1e-6 relative of
    the threshold (oracle fp64 What).  The excused elements are counted and written, with
    their oracle and GPU codes and their distance from the threshold, to a listing file
    named for the case; their number must stay below max(bound_min, bound_frac * n).
    Returns (compared elements, excused elements, mismatches among them)."""
    import os
    import re
    if name is None:
        name = os.environ.get("PYTEST_CURRENT_TEST", "codes").split(" ")[0].split("::")[-1]
    got = np.asarray(got).reshape(-1)
    want = np.asarray(want).reshape(-1)
    gap = np.asarray(gap).reshape(-1)
    band = gap <= NEAR_THRESHOLD
    mism = np.nonzero((got != want) & ~band)[0]
    assert mism.size == 0, f"{name}: {mism.size} code mismatches outside the threshold band (first {mism[:8]})"
    idx = np.nonzero(band)[0]
    flips = int((got[idx] != want[idx]).sum())
    fn = os.path.join(listing_dir(), re.sub(r"[^A-Za-z0-9_.-]+", "_", name) + ".txt")
    with open(fn, "w") as fh:
        fh.write(f"# {name}: {got.size} codes compared, {idx.size} within 1e-6 of the threshold, "
                 f"{flips} of those differ\n# index oracle gpu rel_gap\n")
        for i in idx:
            fh.write(f"{i} {int(want[i])} {int(got[i])} {gap[i]:.3e}\n")
    bound = max(bound_min, int(bound_frac * got.size))
    assert idx.size <= bound, f"{name}: {idx.size} elements in the threshold band (bound {bound})"
    return got.size, int(idx.size), flips
