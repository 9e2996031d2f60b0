"""GPU vs oracle at the workloads' full sizes (the Qwen3-1.7B-, Llama-3-8B- and Qwen3-14B-
shaped blocks with their full calibration batches, and the Qwen3-235B-shaped MoE layer with
all 128 experts), in the launch configuration bench.py times (four-CTA fused forward and
dX, CTA-pair dW), on outputs the fp64 oracle computes one by one.  Samples cover every
output tile of every kernel, and each tile is checked on its own as well as overall:

* group statistics: every group;
* Y and the teacher output: 4 rows of every 512-row M block x 4 columns of every 256-column
  N block, relative Frobenius error per (M block, N block) tile and overall;
* loss and dY: as functions of the GPU's Y and teacher output (the loss over all M x N
  elements in fp64; dY on the sampled entries, per tile);
* dX: the same rows x 4 columns of every 256-column K block, from the GPU's dY (the
  backward's input) and the oracle's Eq. 6 weight, per (M block, K block) tile;
* factor gradients, hard codes and alpha: every group of 2 sampled W rows of every 256-row
  N block, through the oracle's own G = dY^T X for those rows, per (N block, K block) tile
  of the dW kernel; codes outside the threshold band bit-exact, the band listed.
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
    _check_sampled(got, W, X, g, fac, wl.thr_init, phase, s, name=f"full_{wl_name}_{lin_name}_phase{phase}_s{s}")


def _block_sample(n, block, per, r):
    """`per` sorted indices from every `block`-wide block of range(n) (all of a short one)."""
    out = []
    for b0 in range(0, n, block):
        b1 = min(n, b0 + block)
        out.append(np.sort(r.choice(np.arange(b0, b1), min(per, b1 - b0), replace=False)))
    return np.concatenate(out)


def _tile_errs(got, want, rows, cols, rblock, cblock):
    """Relative Frobenius error of every (row block, column block) tile of a sampled
    [len(rows), len(cols)] comparison; returns the worst and its tile."""
    worst, where = 0.0, None
    rb, cb = rows // rblock, cols // cblock
    for a in np.unique(rb):
        for b in np.unique(cb):
            sel = np.ix_(rb == a, cb == b)
            e = U.fro_rel(got[sel], want[sel])
            if e > worst:
                worst, where = e, (int(a), int(b))
    return worst, where


def _check_sampled(got, W, X, g, fac, thr, phase, s, rows_per_block=2, count=None, name=None):
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
    ms = _block_sample(M, 512, 4, r)
    ns = _block_sample(N, 256, 4, r)
    ks = _block_sample(K, 256, 4, r)
    Wq = O.ternary_weight(W, g, stats, fac, phase, s)[0]
    Xs = X[ms].astype(np.float64)
    errs, tiles = {}, {}

    def both(key, a, b, rows, cols, rblock, cblock):
        errs[key] = U.fro_rel(a, b)
        tiles[key] = _tile_errs(a, b, rows, cols, rblock, cblock)

    # forward and teacher forward on the sampled entries
    both("Y", got["Y"][np.ix_(ms, ns)], Xs @ Wq[ns].T, ms, ns, 512, 256)
    both("Y_ref", got["Y_ref"][np.ix_(ms, ns)], Xs @ W[ns].astype(np.float64).T, ms, ns, 512, 256)

    # loss over every element and dY on the sample, from the GPU's own Y and teacher output
    d = got["Y"].astype(np.float64) - got["Y_ref"].astype(np.float64)
    if count is None:
        count = d.size
        loss = float((d * d).sum() / count)
        assert abs(got["loss"] - loss) <= 1e-5 * loss
    both("dY", got["dY"][np.ix_(ms, ns)], 2.0 * d[np.ix_(ms, ns)] / count, ms, ns, 512, 256)
    del d

    # dX from the GPU's dY
    dY = got["dY"].astype(np.float64)
    both("dX", got["dX"][np.ix_(ms, ks)], dY[ms] @ Wq[:, ks], ms, ks, 512, 256)

    # factor gradients, codes and alpha of the sampled rows (all their groups)
    rows = _block_sample(N, 256, rows_per_block, r)
    per_row = K // g
    sub_stats = tuple(_rows(a, rows, per_row) for a in stats)
    sub_fac = tuple(_rows(a, rows, per_row) for a in fac)
    Wsub = W[rows]
    Gsub = dY[:, rows].T @ X.astype(np.float64)
    want = O.factor_grads_from_G(Gsub, Wsub, g, sub_stats, sub_fac, phase, s)
    gcols = np.tile(np.arange(per_row) * g, rows.size).reshape(rows.size, per_row)  # first column of each group
    for nm, w in zip(("g_dmu", "g_dalpha", "g_ddelta"), want):
        a = _rows(got[nm], rows, per_row).reshape(rows.size, per_row)
        b = np.asarray(w).reshape(rows.size, per_row)
        errs[nm] = U.fro_rel(a, b)
        # tiles of the dW kernel: 256 rows of N by 256 columns of K
        worst, where = 0.0, None
        for ab in np.unique(rows // 256):
            for kb in np.unique(gcols[0] // 256):
                sel = np.ix_(rows // 256 == ab, gcols[0] // 256 == kb)
                e = U.fro_rel(a[sel], b[sel])
                if e > worst:
                    worst, where = e, (int(ab), int(kb))
        tiles[nm] = (worst, where)
    print(f"{name or ''} overall {errs} worst tiles {tiles} ({ms.size} x {ns.size} Y samples, "
          f"{rows.size} W rows)")
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, f"tolerance {U.TOL_BF16} exceeded: {bad} (all: {errs})"
    bad = {k: v for k, v in tiles.items() if not v[0] <= U.TOL_BF16}
    assert not bad, f"per-tile tolerance {U.TOL_BF16} exceeded: {bad}"

    T, alpha, gap = O.hard_codes(Wsub, g, sub_stats, sub_fac)
    codes = O.unpack_codes(got["codes"], N * K).reshape(N, K)[rows].reshape(-1)
    U.check_codes(codes, T, gap, name=name)
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
                       rows_per_block=1, count=R * N, name=f"full_moe_expert{e}")
