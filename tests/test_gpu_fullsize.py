"""GPU vs oracle at the benchmark's full size: linears of the Llama-3-8B-shaped block with
M = 8192 token rows, in the launch configuration bench.py times (four-CTA fused forward and
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

WL = "c3_llama3_8b_block"


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


@pytest.mark.parametrize("lin_name,phase,s", [
    ("q_proj", O.PHASE_SOFT, 30.0),       # 4096 -> 4096
    ("k_proj", O.PHASE_HARD, 30.0),       # 4096 -> 1024
    ("gate_proj", O.PHASE_SOFT, 30.0),    # 4096 -> 14336
    ("down_proj", O.PHASE_SOFT, 2.0),     # 14336 -> 4096, two-tanh form
])
def test_c3_full_size_sampled(device, lin_name, phase, s):
    wl = syn.WORKLOADS[WL]
    lin = wl.linear(lin_name)
    M, N, K, g = wl.M, lin.N, lin.K, wl.g
    W = syn.weight(wl, lin)
    X = syn.activations(wl, lin.x, M, K)
    G = N * K // g
    fac = syn.factors(G, 0, f"full/{lin_name}", perturbed=True)
    got = U.gpu_step(W, X, g, fac, wl.thr_init, phase, s, "bf16", device)

    stats = O.group_stats(W, g, wl.thr_init)
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
    loss = float((d * d).sum() / d.size)
    assert abs(got["loss"] - loss) <= 1e-5 * loss
    errs["dY"] = U.fro_rel(got["dY"][np.ix_(ms, ns)], 2.0 * d[np.ix_(ms, ns)] / d.size)
    del d

    # dX from the GPU's dY
    dY = got["dY"].astype(np.float64)
    errs["dX"] = U.fro_rel(got["dX"][np.ix_(ms, ks)], dY[ms] @ Wq[:, ks])

    # factor gradients, codes and alpha of 8 sampled rows (all their groups)
    rows = np.sort(r.choice(N, 8, replace=False))
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
