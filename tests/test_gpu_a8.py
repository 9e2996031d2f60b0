"""GPU vs oracle parity of the 8-bit activation path (W1.58A8, §1 and App. B.2): the
per-token quantizer's codes and scales bit-exact (both sides decide the codes in fp32 with
IEEE division), and the whole A8 calibration step (codes and per-token scales into the
forward, the fused loss against the full-precision teacher, dX straight through the
rounding, dW from the dequantized activations) end to end against the oracle's fp64 step."""
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


@pytest.mark.parametrize("dtype,M,K", [("bf16", 777, 4096), ("bf16", 3, 17408), ("f32", 129, 512)])
def test_act_quant_codes_and_scales(device, dtype, M, K):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(50, f"a8/{dtype}/{M}/{K}")
    X = (r.standard_t(4.0, (M, K)) * r.uniform(0.01, 10.0, (M, 1))).astype(np.float32)
    X[M // 2] = 0.0  # a row of zeros
    if dtype == "bf16":
        X = syn.round_bf16(X)
    Xt = U.to_device(X, dtype, device)
    codes = torch.empty_like(Xt)
    deq = torch.empty_like(Xt)
    scale = torch.empty(M, dtype=torch.float32, device=device)
    C.catq_act_quant_a8(Xt, codes, scale, deq)
    torch.cuda.synchronize()
    q, s = O.act_quant_a8(X)
    np.testing.assert_array_equal(U.to_host(scale), s)
    np.testing.assert_array_equal(U.to_host(codes).astype(np.int64), q)
    want = q * s.astype(np.float64)[:, None]
    assert U.err(U.to_host(deq), want, dtype) <= (3e-3 if dtype == "bf16" else 1e-6)


@pytest.mark.parametrize("wl_name,lin_name,M", [
    ("c2_qwen3_1p7b_block", "q_proj", 300),     # 1% outlier channels x30
    ("c3_llama3_8b_block", "v_proj", 1100),     # Student-t activations, four-CTA clusters
    ("c4_qwen3_14b_block", "k_proj", 700),      # 0.5% outlier channels x50
])
@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 30.0), (O.PHASE_HARD, 30.0)])
def test_a8_step_bf16(device, wl_name, lin_name, M, phase, s):
    wl = syn.WORKLOADS[wl_name]
    lin = wl.linear(lin_name)
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, f"a8/{wl_name}/{lin_name}", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "bf16", device, fused=True, a8=True)
    stats = O.group_stats(W, wl.g, wl.thr_init)
    ref = O.a8_calibration_step(X, W, wl.g, stats, fac, phase, s)
    np.testing.assert_array_equal(got["a8_codes"].astype(np.int64), ref["q"])
    np.testing.assert_array_equal(got["a8_scale"], ref["scale"])
    errs = {k: U.fro_rel(got[k], ref[k]) for k in ("Y_ref", "Y", "dY", "dX", "g_dmu", "g_dalpha", "g_ddelta")}
    errs["loss"] = abs(got["loss"] - ref["loss"]) / ref["loss"]
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, f"tolerance exceeded: {bad} (all: {errs})"


@pytest.mark.parametrize("fused", [False, True])
def test_a8_step_fp32(device, fused):
    wl = syn.WORKLOADS["c1_fp32_linear_512"]
    lin = wl.linears[0]
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, wl.M, lin.K)
    fac = syn.factors(lin.N * lin.K // wl.g, 0, "a8/c1", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, O.PHASE_SOFT, 15.0, "f32", device, fused=fused, a8=True)
    stats = O.group_stats(W, wl.g, wl.thr_init)
    ref = O.a8_calibration_step(X, W, wl.g, stats, fac, O.PHASE_SOFT, 15.0)
    errs = {k: U.max_rel(got[k], ref[k]) for k in ("Y_ref", "Y", "dY", "dX", "g_dmu", "g_dalpha", "g_ddelta")}
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_F32}
    assert not bad, f"tolerance exceeded: {bad} (all: {errs})"
