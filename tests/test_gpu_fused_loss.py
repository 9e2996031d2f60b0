"""GPU vs oracle parity of the fused forward + loss call (catq_soft_ternary_linear_fwd_loss
and its grouped form): the Eq. 7 loss and dY formed in the forward's epilogue from the fp32
accumulator, then the backward from that dY, compared end to end with the oracle's fp64
calibration step (fp32 max relative error 1e-5; bf16 relative Frobenius error 2e-2; codes
bit-exact outside the 1e-6 threshold band).  Also: the extended forward's fp32 output, an
fp32 teacher, a ragged column count, one token row, the sum reduction, and the grouped call.
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


def _compare(got, W, X, g, fac, thr, phase, s, dtype, reduction=0):
    stats = O.group_stats(W, g, thr)
    ref = O.calibration_step(X, W, g, stats, fac, phase, s, reduction=reduction)
    t = U.tol(dtype)
    errs = {k: U.err(got[k], ref[k], dtype) for k in ("Y_ref", "Y", "dY", "dX", "g_dmu", "g_dalpha", "g_ddelta")}
    errs["loss"] = abs(got["loss"] - ref["loss"]) / ref["loss"]
    bad = {k: v for k, v in errs.items() if not v <= t}
    assert not bad, f"tolerance {t} exceeded: {bad} (all: {errs})"
    T, alpha, gap = O.hard_codes(W, g, stats, fac)
    U.check_codes(O.unpack_codes(got["codes"], W.size), T, gap)
    return errs


CASES = [
    ("c2_qwen3_1p7b_block", "q_proj", 300),     # single-CTA tiles, ragged tail
    ("c3_llama3_8b_block", "v_proj", 1100),     # four-CTA clusters, ragged tail
    ("c4_qwen3_14b_block", "k_proj", 700),      # CTA pairs
    ("c3_llama3_8b_block", "down_proj", 520),   # K = 14336, CTA pairs, 8-row tail
]


@pytest.mark.parametrize("wl_name,lin_name,M", CASES)
@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 30.0), (O.PHASE_SOFT, 0.625), (O.PHASE_HARD, 30.0)])
def test_fused_step_bf16(device, wl_name, lin_name, M, phase, s):
    wl = syn.WORKLOADS[wl_name]
    lin = wl.linear(lin_name)
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, f"fused/{wl_name}/{lin_name}", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "bf16", device, fused=True)
    _compare(got, W, X, wl.g, fac, wl.thr_init, phase, s, "bf16")


@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 30.0), (O.PHASE_HARD, 30.0)])
def test_fused_step_fp32(device, phase, s):
    wl = syn.WORKLOADS["c1_fp32_linear_512"]
    lin = wl.linears[0]
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, wl.M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, "fused/c1", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "f32", device, fused=True)
    _compare(got, W, X, wl.g, fac, wl.thr_init, phase, s, "f32")


@pytest.mark.parametrize("teacher_f32", [False, True])
def test_fused_ragged_columns_and_rows(device, teacher_f32):
    """N = 328 leaves 8 columns of the last 16-column epilogue chunk outside the layer; M = 777
    a ragged row tail; the teacher in bf16 and in fp32."""
    N, K, g, M = 328, 384, 128, 777
    r = syn.rng(40, "fused/ragged")
    W = syn.round_bf16((r.standard_normal((N, K)) * 0.02).astype(np.float32))
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 40, "fused/ragged", perturbed=True)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 15.0, "bf16", device, fused=True,
                     teacher_f32=teacher_f32)
    errs = _compare(got, W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 15.0, "bf16")
    if teacher_f32:
        # Y is never rounded before the difference and the teacher not at all: dY carries only
        # its own bf16 rounding
        assert errs["dY"] < 4e-3, errs


def test_fused_sum_reduction_single_row(device):
    N, K, g, M = 256, 256, 128, 1
    r = syn.rng(41, "fused/single")
    W = syn.round_bf16((r.standard_normal((N, K)) * 0.02).astype(np.float32))
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 41, "fused/single", perturbed=True)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16", device, fused=True, reduction=1)
    _compare(got, W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16", reduction=1)


def test_fused_matches_the_two_call_path(device):
    """The fused call and forward + catq_recon_loss agree to the bf16 rounding of Y that the
    two-call path adds (loss to 1e-3, dY to 1e-2)."""
    wl = syn.WORKLOADS["c3_llama3_8b_block"]
    lin = wl.linear("q_proj")
    M = 1100
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, "fused/two-call", perturbed=True)
    a = U.gpu_step(W, X, wl.g, fac, wl.thr_init, O.PHASE_SOFT, 30.0, "bf16", device, fused=True)
    b = U.gpu_step(W, X, wl.g, fac, wl.thr_init, O.PHASE_SOFT, 30.0, "bf16", device, fused=False)
    assert abs(a["loss"] - b["loss"]) <= 1e-3 * b["loss"]
    assert U.fro_rel(a["dY"], b["dY"]) <= 1e-2
    np.testing.assert_array_equal(a["Y"], b["Y"])  # the same accumulator, rounded once


def test_fwd_ex_fp32_output_and_row_scale(device):
    """The extended forward: an fp32 output of a bf16 layer (the accumulator unrounded; fp32
    bound 1e-5 against fp64), and a per-row scale applied to it."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = syn.WORKLOADS["c4_qwen3_14b_block"]
    lin = wl.linear("o_proj")
    M = 600
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, lin.K)
    G = lin.N * lin.K // wl.g
    fac = syn.factors(G, 0, "fused/fwd_ex", perturbed=True)
    layer = C.Layer.create(U.to_device(W, "bf16", device), wl.g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer, wl.thr_init)
    Xt = U.to_device(X, "bf16", device)
    Y32 = torch.empty(M, lin.N, dtype=torch.float32, device=device)
    C.catq_soft_ternary_linear_fwd_ex(layer, C.schedule(C.PHASE_TEACHER), Xt, Y32)
    rs = torch.from_numpy(syn.rng(42, "rs").uniform(0.5, 2.0, M).astype(np.float32)).to(device)
    Ys = torch.empty(M, lin.N, dtype=torch.bfloat16, device=device)
    C.catq_soft_ternary_linear_fwd_ex(layer, C.schedule(C.PHASE_SOFT, 30.0), Xt, Ys, x_row_scale=rs)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    assert U.max_rel(U.to_host(Y32), X.astype(np.float64) @ W.astype(np.float64).T) <= U.TOL_F32
    stats = O.group_stats(W, wl.g, wl.thr_init)
    Wq = O.ternary_weight(W, wl.g, stats, fac, O.PHASE_SOFT, 30.0)[0]
    want = (X.astype(np.float64) @ Wq.T) * U.to_host(rs).astype(np.float64)[:, None]
    assert U.fro_rel(U.to_host(Ys), want) <= U.TOL_BF16


def test_grouped_fused_loss(device):
    """The grouped call's loss over every routed row and its dY, expert by expert against the
    oracle, with the layer-wide element count in the mean."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = dataclasses.replace(syn.WORKLOADS["c5_qwen3_235b_moe"], experts=6, top_k=2, tokens=300)
    lin = wl.linear("gate_proj")
    E, N, K, g = wl.experts, lin.N, lin.K, wl.g
    phase, s = O.PHASE_SOFT, 30.0
    token_of_row, off = syn.moe_routing(wl, seed=3)
    R = int(off[-1])
    W = np.stack([syn.weight(wl, lin, expert=e) for e in range(E)])
    X = syn.activations(wl, lin.x, wl.tokens, K)[token_of_row]
    G = N * K // g
    fac = syn.factors(E * G, 3, "fused/moe", perturbed=True)
    Wt = U.to_device(W.reshape(E * N, K), "bf16", device).reshape(E, N, K)
    layer = C.GroupedLayer.create(Wt, g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer.dense)
    Xt = U.to_device(X, "bf16", device)
    Yref = torch.empty(R, N, dtype=torch.bfloat16, device=device)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), Xt, off, Yref)
    Y = torch.empty_like(Yref)
    dY = torch.empty_like(Yref)
    loss = torch.zeros(1, device=device)
    ws = C.workspace(C.catq_grouped_fwd_loss_workspace_bytes(layer, off), device)
    C.catq_grouped_soft_ternary_linear_fwd_loss(layer, C.schedule(phase, s), Xt, off, Yref, loss, dY, Y=Y,
                                                workspace=ws)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    Yh, dYh, Yrh = U.to_host(Y), U.to_host(dY), U.to_host(Yref).astype(np.float64)
    Yfull = np.zeros((R, N))
    for e in range(E):
        r0, r1 = int(off[e]), int(off[e + 1])
        if r1 == r0:
            continue
        st = O.group_stats(W[e], g)
        Wq = O.ternary_weight(W[e], g, st, tuple(f[e * G:(e + 1) * G] for f in fac), phase, s)[0]
        Yfull[r0:r1] = X[r0:r1].astype(np.float64) @ Wq.T
        assert U.fro_rel(Yh[r0:r1], Yfull[r0:r1]) <= U.TOL_BF16, e
    ref_loss, ref_dY = O.recon_loss(Yfull, Yrh)
    assert abs(loss.item() - ref_loss) <= U.TOL_BF16 * ref_loss
    assert U.fro_rel(dYh, ref_dY) <= U.TOL_BF16
