"""GPU vs oracle parity of the W ~ alpha T + mu reconstruction (the variant of the tab:mu
ablation): Wq = alpha T + mu, dWq/dmu = 1 - f', and inference adding mu times each group's
activation sum.  The same step, tolerances and code checks as the W ~ alpha T parity tests,
with the oracle's with_mu forms as the reference, end to end: every output, the backward's
included, against the oracle's fp64 chain from the same inputs.  The step forms the loss and
dY in the forward's epilogue from the fp32 accumulator (catq_soft_ternary_linear_fwd_loss):
with mu the factor gradient of d_mu carries the plain group sum of G, which projects any
rounding of Y - Y_ref onto the group's activation sums, so Y is not rounded before the
difference."""
import dataclasses

import numpy as np
import pytest

from oracle import catq_oracle as O
from paper_2606_26650_gb300 import synthetic as syn
from tests import gpu_util as U

pytestmark = pytest.mark.gpu

RECON_MU = 1


@pytest.fixture(scope="module")
def device():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.device("cuda:0")


def _compare(got, W, X, g, fac, thr, phase, s, dtype):
    stats = O.group_stats(W, g, thr)
    ref = O.calibration_step(X, W, g, stats, fac, phase, s, with_mu=True)
    t = U.tol(dtype)
    errs = {k: U.err(got[k], ref[k], dtype)
            for k in ("Y_ref", "Y", "dY", "dX", "g_dmu", "g_dalpha", "g_ddelta")}
    errs["loss"] = abs(got["loss"] - ref["loss"]) / ref["loss"]
    print(f"end-to-end errors: {errs}")
    bad = {k: v for k, v in errs.items() if not v <= t}
    assert not bad, f"tolerance {t} exceeded: {bad} (all: {errs})"
    # the deployed form: the same codes and alpha as without mu, plus mu per group
    T, alpha, gap = O.hard_codes(W, g, stats, fac)
    codes = O.unpack_codes(got["codes"], W.size)
    U.check_codes(codes, T, gap)
    np.testing.assert_allclose(got["alpha"], alpha, rtol=2e-6)
    mu = O.modulation(*stats, *fac)[0]
    np.testing.assert_allclose(got["mu"], mu, rtol=1e-5, atol=1e-6 * np.abs(W).max())
    return errs


@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 0.625), (O.PHASE_SOFT, 30.0), (O.PHASE_HARD, 30.0)])
def test_mu_fp32(device, phase, s):
    wl = syn.WORKLOADS["c1_fp32_linear_512"]
    lin = wl.linears[0]
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, wl.M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, "mu/c1", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "f32", device, recon=RECON_MU, fused=True)
    _compare(got, W, X, wl.g, fac, wl.thr_init, phase, s, "f32")


@pytest.mark.parametrize("wl_name,lin_name,M", [
    ("c2_qwen3_1p7b_block", "q_proj", 300),     # 1-CTA tiles, ragged tail
    ("c3_llama3_8b_block", "v_proj", 1100),     # 2-CTA tiles over 3 tiles, ragged tail
    ("c4_qwen3_14b_block", "k_proj", 700),
])
@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 30.0), (O.PHASE_SOFT, 0.625), (O.PHASE_HARD, 30.0)])
def test_mu_bf16(device, wl_name, lin_name, M, phase, s):
    wl = syn.WORKLOADS[wl_name]
    lin = wl.linear(lin_name)
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, f"mu/{wl_name}/{lin_name}", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "bf16", device, recon=RECON_MU, fused=True)
    _compare(got, W, X, wl.g, fac, wl.thr_init, phase, s, "bf16")


@pytest.mark.parametrize("teacher_f32", [False, True])
def test_mu_bf16_ragged_and_offset_groups(device, teacher_f32):
    """A ragged shape whose groups carry a large common offset, where alpha T alone misses
    most of W and mu carries it; end to end with the teacher output in bf16 and in fp32."""
    N, K, g, M = 328, 384, 128, 777
    r = syn.rng(6, "mu/ragged")
    off = np.repeat(r.uniform(-0.05, 0.05, N * K // g), g).reshape(N, K)
    W = syn.round_bf16((r.standard_normal((N, K)) * 0.02 + off).astype(np.float32))
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 6, "mu/ragged", perturbed=True)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 15.0, "bf16", device, recon=RECON_MU, fused=True,
                     teacher_f32=teacher_f32)
    _compare(got, W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 15.0, "bf16")


def test_mu_degenerate_groups(device):
    """Constant groups (alpha0 = 0) reconstruct as their value mu0 and get zero factor
    gradients."""
    r = syn.rng(7, "mu/degenerate")
    N, K, g, M = 64, 256, 128, 64
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    W[::3, :g] = np.float32(0.0078125)
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 7, "mu/degenerate", perturbed=False)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16", device, recon=RECON_MU, fused=True)
    dead = np.arange(0, N, 3) * (K // g)
    assert not got["g_dmu"][dead].any() and not got["g_dalpha"][dead].any()
    _compare(got, W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16")


def test_mu_modulate_ternarize(device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = syn.WORKLOADS["c3_llama3_8b_block"]
    lin = wl.linear("k_proj")
    W = syn.weight(wl, lin)
    G = lin.N * lin.K // wl.g
    fac = syn.factors(G, 0, "mu/modulate", perturbed=True)
    stats = O.group_stats(W, wl.g)
    layer = C.Layer.create(U.to_device(W, "bf16", device), wl.g, *(torch.from_numpy(f).to(device) for f in fac),
                           recon=RECON_MU)
    C.catq_group_stats(layer)
    for phase, s in ((O.PHASE_SOFT, 0.625), (O.PHASE_SOFT, 30.0), (O.PHASE_HARD, 30.0), (O.PHASE_TEACHER, 0.0)):
        Wq = torch.empty_like(layer.W)
        C.catq_modulate_ternarize(layer, C.schedule(phase, s), Wq)
        torch.cuda.synchronize()
        Wq_ref = O.ternary_weight(W, wl.g, stats, fac, phase, s, with_mu=True)[0]
        assert U.fro_rel(U.to_host(Wq), Wq_ref) < 1e-2


@pytest.mark.parametrize("N,K,g,B", [
    (8192, 1024, 128, 3),     # four rows per warp
    (4096, 4096, 128, 1),     # two rows per warp
    (520, 192, 64, 8),        # one row per warp, ragged N
    (64, 512, 512, 11),       # channel-wise groups
])
def test_mu_ternary_infer(device, N, K, g, B):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(8, f"mu/infer/{N}/{K}/{g}")
    off = np.repeat(r.uniform(-0.03, 0.03, N * K // g), g).reshape(N, K)
    W = syn.round_bf16((r.standard_normal((N, K)) * 0.02 + off).astype(np.float32))
    X = syn.round_bf16(r.standard_normal((B, K)).astype(np.float32))
    G = N * K // g
    fac = syn.factors(G, 8, f"mu/infer/{N}/{K}", perturbed=True)
    layer = C.Layer.create(U.to_device(W, "bf16", device), g, *(torch.from_numpy(f).to(device) for f in fac),
                           recon=RECON_MU)
    C.catq_group_stats(layer)
    codes = torch.empty(N * K // 4, dtype=torch.uint8, device=device)
    alpha = torch.empty(G, dtype=torch.float32, device=device)
    mu = torch.empty(G, dtype=torch.float32, device=device)
    C.catq_hard_ternarize_pack(layer, codes, alpha, mu)
    Xt = U.to_device(X, "bf16", device)
    Y = torch.empty(B, N, dtype=torch.bfloat16, device=device)
    C.catq_ternary_infer(codes, alpha, N, K, g, Xt, Y, mu=mu)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    want = O.ternary_infer(U.to_host(codes), U.to_host(alpha), N, K, g, X, mu=U.to_host(mu))
    assert U.fro_rel(U.to_host(Y), want) <= U.TOL_BF16
    # and the deployed form reproduces the HARD-phase forward with mu (up to bf16 rounding)
    stats = O.group_stats(W, g)
    Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_HARD, 30.0, with_mu=True)[0]
    assert U.fro_rel(U.to_host(Y), X.astype(np.float64) @ Wq.T) <= U.TOL_BF16


def test_mu_grouped_experts(device):
    """The grouped calls with mu (each expert's operand constants and mu plane at its own
    offset of the [E, 5 G] array), expert by expert against the oracle."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = dataclasses.replace(syn.WORKLOADS["c5_qwen3_235b_moe"], experts=6, top_k=2, tokens=64)
    lin = wl.linear("gate_proj")
    E, N, K, g = wl.experts, lin.N, lin.K, wl.g
    phase, s = O.PHASE_SOFT, 30.0
    token_of_row, off = syn.moe_routing(wl, seed=1)
    R = int(off[-1])
    W = np.stack([syn.weight(wl, lin, expert=e) for e in range(E)])
    X = syn.activations(wl, lin.x, wl.tokens, K)[token_of_row]
    G = N * K // g
    fac = syn.factors(E * G, 1, "mu/moe", perturbed=True)
    Wt = U.to_device(W.reshape(E * N, K), "bf16", device).reshape(E, N, K)
    layer = C.GroupedLayer.create(Wt, g, *(torch.from_numpy(f).to(device) for f in fac), recon=RECON_MU)
    assert layer.dense.op_const.numel() == 5 * E * G
    C.catq_group_stats(layer.dense)
    Xt = U.to_device(X, "bf16", device)
    Y = torch.empty(R, N, dtype=torch.bfloat16, device=device)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(phase, s), Xt, off, Y)
    dY = U.to_device(syn.rng(9, "mu/moe/dY").standard_normal((R, N)).astype(np.float32) * 1e-3, "bf16", device)
    dX = torch.empty_like(Xt)
    gr = [torch.empty(E * G, device=device) for _ in range(3)]
    ws = C.workspace(C.catq_grouped_bwd_workspace_bytes(layer, off), device)
    C.catq_grouped_soft_ternary_linear_bwd(layer, C.schedule(phase, s), Xt, dY, off, dX, *gr, ws)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    Yh, dXh, dYh = U.to_host(Y), U.to_host(dX), U.to_host(dY).astype(np.float64)
    grh = [U.to_host(t) for t in gr]
    for e in range(E):
        r0, r1 = int(off[e]), int(off[e + 1])
        gs = slice(e * G, (e + 1) * G)
        st = O.group_stats(W[e], g)
        fe = tuple(f[gs] for f in fac)
        Wq = O.ternary_weight(W[e], g, st, fe, phase, s, with_mu=True)[0]
        if r1 > r0:
            assert U.fro_rel(Yh[r0:r1], X[r0:r1].astype(np.float64) @ Wq.T) <= U.TOL_BF16
            assert U.fro_rel(dXh[r0:r1], dYh[r0:r1] @ Wq) <= U.TOL_BF16
        want = O.linear_bwd(X[r0:r1], dYh[r0:r1], W[e], g, st, fe, phase, s, with_mu=True)[1:]
        for name, got, w in zip(("g_dmu", "g_dalpha", "g_ddelta"), grh, want):
            if r1 > r0:
                assert U.fro_rel(got[gs], w) <= U.TOL_BF16, (e, name)
            else:
                assert not got[gs].any(), (e, name)
