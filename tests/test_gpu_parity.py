"""GPU vs oracle parity of the whole calibration step, through the C ABI.

Each case runs group statistics, the teacher and phase forwards, the reconstruction loss,
the backward (dX and the three factor gradients) and the hard pack on the GPU, and the
same step in the fp64 oracle from the same seeded inputs, then compares every output
element by element: fp32 within max relative error 1e-5, bf16 within relative Frobenius
error 2e-2, ternary codes bit-exact outside the 1e-6 relative threshold band.
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


def _compare(got, W, X, g, fac, thr, phase, s, dtype):
    stats = O.group_stats(W, g, thr)
    ref = O.calibration_step(X, W, g, stats, fac, phase, s)
    # statistics are fp32 roundings of fp64 sums
    np.testing.assert_allclose(got["mu0"], stats[0], rtol=1e-5, atol=1e-7 * np.abs(W).max())
    np.testing.assert_allclose(got["alpha0"], stats[1], rtol=1e-6)
    np.testing.assert_allclose(got["delta0"], stats[2], rtol=1e-6)
    t = U.tol(dtype)
    errs = {k: U.err(got[k], ref[k], dtype) for k in ("Y_ref", "Y", "dY", "g_dmu", "g_dalpha", "g_ddelta")}
    if "dX" in got:
        errs["dX"] = U.err(got["dX"], ref["dX"], dtype)
    errs["loss"] = abs(got["loss"] - ref["loss"]) / ref["loss"]
    bad = {k: v for k, v in errs.items() if not v <= t}
    assert not bad, f"tolerance {t} exceeded: {bad} (all: {errs})"
    T, alpha, gap = O.hard_codes(W, g, stats, fac)
    codes = O.unpack_codes(got["codes"], W.size)
    U.check_codes(codes, T, gap)
    np.testing.assert_allclose(got["alpha"], alpha, rtol=2e-6)
    return errs


# ---------------------------------------------------------------- config 1 (fp32, full size)

@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 0.625), (O.PHASE_SOFT, 15.0), (O.PHASE_SOFT, 30.0),
                                     (O.PHASE_HARD, 30.0)])
@pytest.mark.parametrize("perturbed", [False, True])
def test_c1_fp32_full(device, phase, s, perturbed):
    wl = syn.WORKLOADS["c1_fp32_linear_512"]
    lin = wl.linears[0]
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, wl.M, lin.K)
    G = lin.N * lin.K // wl.g
    fac = syn.factors(G, 0, "c1", perturbed)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "f32", device)
    _compare(got, W, X, wl.g, fac, wl.thr_init, phase, s, "f32")


# ---------------------------------------------------------------- bf16 configs, reduced M

BF16_CASES = [
    # (workload, linear, M): M = 300 runs the 1-CTA tiles with a ragged tail; M = 1100 runs
    # the 2-CTA tiles (512 rows) over 3 tiles with a ragged tail.
    ("c2_qwen3_1p7b_block", "q_proj", 300),
    ("c2_qwen3_1p7b_block", "k_proj", 1100),
    ("c2_qwen3_1p7b_block", "down_proj", 300),
    ("c3_llama3_8b_block", "v_proj", 1100),
    ("c3_llama3_8b_block", "gate_proj", 300),
    ("c4_qwen3_14b_block", "o_proj", 300),
    ("c4_qwen3_14b_block", "k_proj", 700),
]


@pytest.mark.parametrize("wl_name,lin_name,M", BF16_CASES)
@pytest.mark.parametrize("phase,s", [(O.PHASE_SOFT, 30.0), (O.PHASE_SOFT, 0.625), (O.PHASE_HARD, 30.0)])
def test_bf16_reduced(device, wl_name, lin_name, M, phase, s):
    wl = syn.WORKLOADS[wl_name]
    lin = wl.linear(lin_name)
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, lin.K)
    G = lin.N * lin.K // wl.g
    fac = syn.factors(G, 0, f"{wl_name}/{lin_name}", perturbed=True)
    got = U.gpu_step(W, X, wl.g, fac, wl.thr_init, phase, s, "bf16", device)
    _compare(got, W, X, wl.g, fac, wl.thr_init, phase, s, "bf16")


@pytest.mark.parametrize("N,K,g,M", [(328, 384, 128, 777), (64, 512, 512, 96), (520, 192, 64, 1)])
def test_bf16_ragged_shapes(device, N, K, g, M):
    """N not a multiple of the 256-column tile, K not a multiple of 256, channel-wise
    groups (g = K), a single token."""
    r = syn.rng(1, f"ragged/{N}/{K}/{g}/{M}")
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 1, f"ragged/{N}/{K}", perturbed=True)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 15.0, "bf16", device)
    _compare(got, W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 15.0, "bf16")


def test_degenerate_group_bf16(device):
    """Constant groups (alpha0 = 0) produce zero weights, codes 0 and zero gradients."""
    r = syn.rng(2, "degenerate")
    N, K, g, M = 64, 256, 128, 64
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    W[::3, :g] = np.float32(0.0078125)
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    fac = syn.factors(N * K // g, 2, "degenerate", perturbed=False)
    got = U.gpu_step(W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16", device)
    dead = np.arange(0, N, 3) * (K // g)
    assert not got["g_dmu"][dead].any() and not got["g_dalpha"][dead].any()
    _compare(got, W, X, g, fac, O.THR_HALF, O.PHASE_SOFT, 30.0, "bf16")


def test_teacher_bwd_zero_grads(device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(3, "teacher")
    N, K, g, M = 256, 256, 128, 128
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    dY = syn.round_bf16(r.standard_normal((M, N)).astype(np.float32))
    layer = C.Layer.create(U.to_device(W, "bf16", device), g)
    C.catq_group_stats(layer)
    dYt, Xt = U.to_device(dY, "bf16", device), U.to_device(X, "bf16", device)
    dX = torch.empty_like(Xt)
    gr = [torch.full((layer.G,), 7.0, device=device) for _ in range(3)]
    C.catq_soft_ternary_linear_bwd(layer, C.schedule(C.PHASE_TEACHER), Xt, dYt, dX, *gr, None)
    torch.cuda.synchronize()
    assert all(not t.any() for t in gr)
    assert U.fro_rel(U.to_host(dX), dY.astype(np.float64) @ W) < U.TOL_BF16


def test_bwd_deterministic(device):
    """Two backward runs give bit-identical factor gradients (fixed reduction order)."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(4, "determinism")
    N, K, g, M = 1024, 512, 128, 1024
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    X = syn.round_bf16(r.standard_normal((M, K)).astype(np.float32))
    dY = syn.round_bf16(r.standard_normal((M, N)).astype(np.float32) * 1e-3)
    layer = C.Layer.create(U.to_device(W, "bf16", device), g)
    C.catq_group_stats(layer)
    Xt, dYt = U.to_device(X, "bf16", device), U.to_device(dY, "bf16", device)
    ws = C.workspace(C.catq_bwd_workspace_bytes(layer, M), device)
    runs = []
    for _ in range(2):
        gr = [torch.empty(layer.G, device=device) for _ in range(3)]
        C.catq_soft_ternary_linear_bwd(layer, C.schedule(C.PHASE_SOFT, 30.0), Xt, dYt, None, *gr, ws)
        runs.append([t.cpu() for t in gr])
    for a, b in zip(*runs):
        assert torch.equal(a, b)


def test_modulate_ternarize_matches_oracle(device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = syn.WORKLOADS["c3_llama3_8b_block"]
    lin = wl.linear("k_proj")
    W = syn.weight(wl, lin)
    G = lin.N * lin.K // wl.g
    fac = syn.factors(G, 0, "modulate", perturbed=True)
    stats = O.group_stats(W, wl.g)
    layer = C.Layer.create(U.to_device(W, "bf16", device), wl.g,
                           *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer)
    for phase, s in ((O.PHASE_SOFT, 0.625), (O.PHASE_SOFT, 30.0), (O.PHASE_HARD, 30.0), (O.PHASE_TEACHER, 0.0)):
        Wq = torch.empty_like(layer.W)
        T = torch.empty(W.shape, dtype=torch.int8, device=device)
        alpha = torch.empty(G, device=device)
        C.catq_modulate_ternarize(layer, C.schedule(phase, s), Wq, T, alpha)
        torch.cuda.synchronize()
        Wq_ref = O.ternary_weight(W, wl.g, stats, fac, phase, s)[0]
        assert U.fro_rel(U.to_host(Wq), Wq_ref) < 1e-2
        Tr, ar, gap = O.hard_codes(W, wl.g, stats, fac)
        U.check_codes(U.to_host(T).reshape(-1), Tr, gap, name=f"modulate_ternarize_phase{phase}_s{s}")
        np.testing.assert_allclose(U.to_host(alpha), ar, rtol=2e-6)


def test_recon_loss_sum_and_tail(device):
    """Sum reduction, an element count that is not a multiple of the vector width, fp32."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(5, "loss")
    for dtype, n in (("f32", 1000003), ("bf16", 77777)):
        a = r.standard_normal(n).astype(np.float32)
        b = r.standard_normal(n).astype(np.float32)
        if dtype == "bf16":
            a, b = syn.round_bf16(a), syn.round_bf16(b)
        ta, tb = U.to_device(a, dtype, device), U.to_device(b, dtype, device)
        loss = torch.zeros(1, device=device)
        dY = torch.empty_like(ta)
        ws = C.workspace(C.catq_recon_loss_workspace_bytes(n), device)
        C.catq_recon_loss(ta, tb, loss, dY, ws, reduction=C.REDUCE_SUM)
        torch.cuda.synchronize()
        ref_loss, ref_dy = O.recon_loss(a, b, 1)
        assert abs(loss.item() - ref_loss) / ref_loss < 1e-6
        assert U.err(U.to_host(dY), ref_dy, dtype) < U.tol(dtype)
