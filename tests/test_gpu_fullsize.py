"""GPU vs oracle at the workloads' full sizes (the Qwen3-1.7B-, Llama-3-8B- and Qwen3-14B-
shaped blocks with their full calibration batches, and the Qwen3-235B-shaped MoE layer with
all 128 experts), in the launch configuration bench.py times (four-CTA fused forward and
dX, CTA-pair dW), on outputs the fp64 oracle computes one by one.

* group statistics: every group;
* Y and the teacher output: a 64 x 64 sample of rows and columns;
* loss and dY: as functions of the GPU's Y and teacher output (the loss over all M x N
  elements in fp64; dY on the sampled entries);
* dX: a 64 x 64 sample, from the GPU's dY (the backward's input) and the oracle's Eq. 6
  weight;
* factor gradients, hard codes and alpha: every group of 8 sampled W rows, through the
  oracle's own G = dY^T X for those rows.
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


def _rows(a, rows, per_row):
    """The per-group entries of W rows `rows` (groups are runs of g inside a row)."""
    a = np.asarray(a)
    return a.reshape(-1, per_row)[rows].reshape(-1)


@pytest.mark.parametrize("wl_name,lin_name,phase,s", [
    ("c3_llama3_8b_block", "q_proj", O.PHASE_SOFT, 30.0),       # 4096 -> 4096 (the bench config)
    ("c3_llama3_8b_block", "k_proj", O.PHASE_HARD, 30.0),       # 4096 -> 1024
    ("c3_llama3_8b_block", "gate_proj", O.PHASE_SOFT, 30.0),    # 4096 -> 14336
    ("c3_llama3_8b_block", "down_proj", O.PHASE_SOFT, 2.0),     # 14336 -> 4096, two-tanh form
    ("c2_qwen3_1p7b_block", "up_proj", O.PHASE_SOFT, 30.0),     # 2048 -> 6144, outlier channels
    ("c4_qwen3_14b_block", "gate_proj", O.PHASE_SOFT, 30.0),    # 5120 -> 17408, M = 4096
    ("c4_qwen3_14b_block", "down_proj", O.PHASE_HARD, 30.0),    # 17408 -> 5120
])
def test_block_full_size_sampled(device, wl_name, lin_name, phase, s):
    wl = syn.WORKLOADS[wl_name]
    lin = wl.linear(lin_name)
    M, N, K, g = wl.M, lin.N, lin.K, wl.g
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, K)
    G = N * K // g
    fac = syn.factors(G, 0, f"full/{wl_name}/{lin_name}", perturbed=True)
    got = U.gpu_step(W, X, g, fac, wl.thr_init, phase, s, "bf16", device)
    _check_sampled(got, W, X, g, fac, wl.thr_init, phase, s, rows_sampled=8)


def _check_sampled(got, W, X, g, fac, thr, phase, s, rows_sampled, count=None):
    """The checks of the module docstring for one dense layer (all arrays on the host).
    `count`: the loss's element count when the rows are part of a larger batch (the loss
    itself is then checked by the caller)."""
    M, K = X.shape
    N = W.shape[0]

    stats = O.group_stats(W, g, thr)
    np.testing.assert_allclose(got["mu0"], stats[0], rtol=1e-5, atol=1e-7 * np.abs(W).max())
    np.testing.assert_allclose(got["alpha0"], stats[1], rtol=1e-6)
    np.testing.assert_allclose(got["delta0"], stats[2], rtol=1e-6)

    r = np.random.default_rng(7)
    ms = np.sort(r.choice(M, 64, replace=False))
    ns = np.sort(r.choice(N, 64, replace=False))
    ks = np.sort(r.choice(K, 64, replace=False))
    Wq = O.ternary_weight(W, g, stats, fac, phase, s)[0]
    Xs = X[ms].astype(np.float64)

    # forward and teacher forward on the sampled entries
    errs = {"Y": U.fro_rel(got["Y"][np.ix_(ms, ns)], Xs @ Wq[ns].T),
            "Y_ref": U.fro_rel(got["Y_ref"][np.ix_(ms, ns)], Xs @ W[ns].astype(np.float64).T)}

    # loss over every element and dY on the sample, from the GPU's own Y and teacher output
    d = got["Y"].astype(np.float64) - got["Y_ref"].astype(np.float64)
    if count is None:
        count = d.size
        loss = float((d * d).sum() / count)
        assert abs(got["loss"] - loss) <= 1e-5 * loss
    errs["dY"] = U.fro_rel(got["dY"][np.ix_(ms, ns)], 2.0 * d[np.ix_(ms, ns)] / count)
    del d

    # dX from the GPU's dY
    dY = got["dY"].astype(np.float64)
    errs["dX"] = U.fro_rel(got["dX"][np.ix_(ms, ks)], dY[ms] @ Wq[:, ks])

    # factor gradients, codes and alpha of 8 sampled rows (all their groups)
    rows = np.sort(r.choice(N, rows_sampled, replace=False))
    per_row = K // g
    sub_stats = tuple(_rows(a, rows, per_row) for a in stats)
    sub_fac = tuple(_rows(a, rows, per_row) for a in fac)
    Wsub = W[rows]
    Gsub = dY[:, rows].T @ X.astype(np.float64)
    want = O.factor_grads_from_G(Gsub, Wsub, g, sub_stats, sub_fac, phase, s)
    for name, w in zip(("g_dmu", "g_dalpha", "g_ddelta"), want):
        errs[name] = U.fro_rel(_rows(got[name], rows, per_row), w)
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, f"tolerance {U.TOL_BF16} exceeded: {bad} (all: {errs})"

    T, alpha, gap = O.hard_codes(Wsub, g, sub_stats, sub_fac)
    codes = O.unpack_codes(got["codes"], N * K).reshape(N, K)[rows].reshape(-1)
    mism = np.nonzero((codes != T) & (gap > U.NEAR_THRESHOLD))[0]
    assert mism.size == 0, f"{mism.size} code mismatches outside the threshold band"
    np.testing.assert_allclose(_rows(got["alpha"], rows, per_row), alpha, rtol=2e-6)


def test_c5_moe_full_size_sampled(device):
    """All 128 experts of the MoE layer's gate_proj with top-8 Zipf(1.1) routing of 8192
    tokens (65,536 routed rows) through the grouped calls; the most and least loaded experts
    and a median one are checked like a dense layer on their own rows."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    wl = syn.WORKLOADS["c5_qwen3_235b_moe"]
    lin = wl.linear("gate_proj")
    E, N, K, g = wl.experts, lin.N, lin.K, wl.g
    phase, s = O.PHASE_SOFT, 30.0
    token_of_row, off = syn.moe_routing(wl, seed=0)
    R = int(off[-1])
    assert R == wl.tokens * wl.top_k
    counts = np.diff(off)
    W = np.stack([syn.weight(wl, lin, expert=e) for e in range(E)])
    X_tok = syn.activations(wl, lin.x, wl.tokens, K)
    G = N * K // g
    fac = syn.factors(E * G, 0, "full/moe/gate_proj", perturbed=True)

    Wt = U.to_device(W.reshape(E * N, K), "bf16", device).reshape(E, N, K)
    layer = C.GroupedLayer.create(Wt, g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer.dense, wl.thr_init)
    Xt = U.to_device(X_tok, "bf16", device)[torch.from_numpy(token_of_row).to(device)]
    Yref = torch.empty(R, N, dtype=torch.bfloat16, device=device)
    Y = torch.empty_like(Yref)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), Xt, off, Yref)
    C.catq_grouped_soft_ternary_linear_fwd(layer, C.schedule(phase, s), Xt, off, Y)
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    dY = torch.empty_like(Y)
    C.catq_recon_loss(Y, Yref, loss, dY, C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), device))
    dX = torch.empty_like(Xt)
    gr = [torch.empty(E * G, dtype=torch.float32, device=device) for _ in range(3)]
    ws = C.workspace(C.catq_grouped_bwd_workspace_bytes(layer, off), device)
    C.catq_grouped_soft_ternary_linear_bwd(layer, C.schedule(phase, s), Xt, dY, off, dX, *gr, workspace=ws)
    codes = torch.empty(E * N * K // 4, dtype=torch.uint8, device=device)
    alpha = torch.empty(E * G, dtype=torch.float32, device=device)
    C.catq_hard_ternarize_pack(layer.dense, codes, alpha)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0

    order = np.argsort(counts)
    nonempty = order[counts[order] > 0]
    experts = sorted({int(order[-1]), int(nonempty[0]), int(order[len(order) // 2])})
    host = {k: U.to_host(v) for k, v in dict(Y=Y, Y_ref=Yref, dY=dY, dX=dX, mu0=layer.dense.mu0,
                                             alpha0=layer.dense.alpha0, delta0=layer.dense.delta0,
                                             g0=gr[0], g1=gr[1], g2=gr[2], alpha=alpha).items()}
    codes_h = U.to_host(codes)
    d = host["Y"].astype(np.float64) - host["Y_ref"].astype(np.float64)
    want_loss = float((d * d).sum() / d.size)
    assert abs(float(loss.item()) - want_loss) <= 1e-5 * want_loss
    del d
    for e in experts:
        r0, r1 = int(off[e]), int(off[e + 1])
        gs = slice(e * G, (e + 1) * G)
        # the expert's rows of the batch against the expert alone; the loss is the layer's, so
        # each expert's dY keeps the layer-wide scale (R N elements).
        got = dict(Y=host["Y"][r0:r1], Y_ref=host["Y_ref"][r0:r1], dY=host["dY"][r0:r1], dX=host["dX"][r0:r1],
                   mu0=host["mu0"][gs], alpha0=host["alpha0"][gs], delta0=host["delta0"][gs],
                   g_dmu=host["g0"][gs], g_dalpha=host["g1"][gs], g_ddelta=host["g2"][gs],
                   alpha=host["alpha"][gs], codes=codes_h[e * N * K // 4:(e + 1) * N * K // 4])
        _check_sampled(got, W[e], X_tok[token_of_row[r0:r1]], g, tuple(f[gs] for f in fac), wl.thr_init, phase, s,
                       rows_sampled=4, count=R * N)
