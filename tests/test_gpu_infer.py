"""GPU parity of inference with the deployed form (codes + group scales, App. B.2): the
codes and alpha come from catq_hard_ternarize_pack on the GPU (whose parity with the oracle
test_gpu_parity checks), and catq_ternary_infer's Y is compared with the oracle's
ternary_infer on the same codes, alpha and X (bf16 relative Frobenius error 2e-2)."""
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


@pytest.mark.parametrize("N,K,g,B", [
    (1024, 4096, 128, 1),     # decode, one token row
    (1024, 4096, 128, 3),
    (520, 192, 64, 8),        # ragged N, a single full pass of 8 rows
    (64, 512, 512, 11),       # channel-wise groups, two passes (8 + 3)
    (4096, 14336, 128, 2),    # the Llama-3-8B-shaped down_proj
    (328, 1024, 128, 5),      # a partial 128-row block, K split over two CTAs
    (256, 2048, 128, 19),     # two passes over 16 token rows
])
def test_ternary_infer_matches_oracle(device, N, K, g, B):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(5, f"infer/{N}/{K}/{g}")
    W = syn.round_bf16(r.standard_normal((N, K)).astype(np.float32) * 0.02)
    X = syn.round_bf16(r.standard_normal((B, K)).astype(np.float32))
    G = N * K // g
    fac = syn.factors(G, 5, f"infer/{N}/{K}", perturbed=True)
    layer = C.Layer.create(U.to_device(W, "bf16", device), g, *(torch.from_numpy(f).to(device) for f in fac))
    C.catq_group_stats(layer)
    codes = torch.empty(N * K // 4, dtype=torch.uint8, device=device)
    alpha = torch.empty(G, dtype=torch.float32, device=device)
    C.catq_hard_ternarize_pack(layer, codes, alpha)
    Xt = U.to_device(X, "bf16", device)
    Y = torch.empty(B, N, dtype=torch.bfloat16, device=device)
    for _ in range(2):  # twice: the result does not depend on earlier calls
        C.catq_ternary_infer(codes, alpha, N, K, g, Xt, Y)
        torch.cuda.synchronize()
        assert C.catq_device_status() == 0
        want = O.ternary_infer(U.to_host(codes), U.to_host(alpha), N, K, g, X)
        assert U.fro_rel(U.to_host(Y), want) <= U.TOL_BF16


@pytest.mark.parametrize("shapes,g,B,with_mu", [
    # the q, k, v projections of the Llama-3-8B-shaped block, one token row
    (((4096, 4096), (1024, 4096), (1024, 4096)), 128, 1, False),
    # gate and up, then a down-shaped layer with K = 14336 (several slabs) in the same launch
    (((14336, 4096), (14336, 4096), (4096, 14336)), 128, 8, False),
    # ragged row counts, two token blocks (8 + 3), the W ~ alpha T + mu form
    (((520, 192), (328, 1024), (64, 192)), 64, 11, True),
])
def test_ternary_infer_batched_matches_oracle(device, shapes, g, B, with_mu):
    """Several independent layers in one launch: each layer's Y against the oracle on its own
    codes, scales and X."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    layers, want = [], []
    for i, (N, K) in enumerate(shapes):
        r = syn.rng(6, f"infer_batched/{i}/{N}/{K}")
        off = np.repeat(r.uniform(-0.03, 0.03, N * K // g), g).reshape(N, K) if with_mu else 0.0
        W = syn.round_bf16((r.standard_normal((N, K)) * 0.02 + off).astype(np.float32))
        X = syn.round_bf16(r.standard_normal((B, K)).astype(np.float32))
        G = N * K // g
        fac = syn.factors(G, 6, f"infer_batched/{i}", perturbed=True)
        layer = C.Layer.create(U.to_device(W, "bf16", device), g, *(torch.from_numpy(f).to(device) for f in fac),
                               recon=1 if with_mu else 0)
        C.catq_group_stats(layer)
        codes = torch.empty(N * K // 4, dtype=torch.uint8, device=device)
        alpha = torch.empty(G, dtype=torch.float32, device=device)
        mu = torch.empty(G, dtype=torch.float32, device=device) if with_mu else None
        C.catq_hard_ternarize_pack(layer, codes, alpha, mu)
        Xt = U.to_device(X, "bf16", device)
        Y = torch.empty(B, N, dtype=torch.bfloat16, device=device)
        layers.append((codes, alpha, N, K, Xt, Y, mu))
        want.append((X, N, K))
    for _ in range(2):
        C.catq_ternary_infer_batched(layers, g)
        torch.cuda.synchronize()
        assert C.catq_device_status() == 0
        for (codes, alpha, N, K, Xt, Y, mu), (X, _, _) in zip(layers, want):
            ref = O.ternary_infer(U.to_host(codes), U.to_host(alpha), N, K, g, X,
                                  mu=U.to_host(mu) if mu is not None else None)
            assert U.fro_rel(U.to_host(Y), ref) <= U.TOL_BF16, (N, K)


def _packed_layer(device, N, K, g, tag, with_mu=False):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(7, f"infer_staged/{tag}/{N}/{K}")
    off = np.repeat(r.uniform(-0.03, 0.03, N * K // g), g).reshape(N, K) if with_mu else 0.0
    W = syn.round_bf16((r.standard_normal((N, K)) * (1.0 / np.sqrt(K)) + off).astype(np.float32))
    G = N * K // g
    fac = syn.factors(G, 7, f"infer_staged/{tag}", perturbed=True)
    layer = C.Layer.create(U.to_device(W, "bf16", device), g, *(torch.from_numpy(f).to(device) for f in fac),
                           recon=1 if with_mu else 0)
    C.catq_group_stats(layer)
    codes = torch.empty(N * K // 4, dtype=torch.uint8, device=device)
    alpha = torch.empty(G, dtype=torch.float32, device=device)
    mu = torch.empty(G, dtype=torch.float32, device=device) if with_mu else None
    C.catq_hard_ternarize_pack(layer, codes, alpha, mu)
    return codes, alpha, mu


# (N, K, index of the layer whose Y is this layer's X, or -1 for the launch input), per stage
CHAIN = [
    [(1024, 512, -1)],
    [(768, 1024, 0), (512, 1024, 0)],     # two independent readers of stage 0
    [(1024, 768, 1)],
    [(512, 1024, 3), (512, 512, 2)],      # readers of stage 2 and of stage 1
]


@pytest.mark.parametrize("B,with_mu", [(1, False), (8, False), (11, True)])
def test_ternary_infer_staged_chain(device, B, with_mu):
    """A chain of dependent layers in one cooperative launch: each layer's Y against the oracle
    on its own codes and scales and on the X the launch gave it (the Y of an earlier stage, read
    back), so a layer that read its X before the producing stage finished would fail.  Outputs
    are filled with NaN first; the sync buffer is zero after every call, and a second call
    gives bit-identical outputs."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    g = 128
    x0 = U.to_device(syn.round_bf16(syn.rng(8, "infer_staged/x0").standard_normal((B, 512)).astype(np.float32)),
                     "bf16", device)
    layers, stages, ys = [], [], []
    for s, stage in enumerate(CHAIN):
        for N, K, src in stage:
            codes, alpha, mu = _packed_layer(device, N, K, g, f"{s}/{len(layers)}", with_mu)
            X = x0 if src < 0 else ys[src]
            assert X.shape[1] == K
            Y = torch.full((B, N), float("nan"), dtype=torch.bfloat16, device=device)
            layers.append((codes, alpha, N, K, X, Y, mu))
            stages.append(s)
            ys.append(Y)
    sync = torch.zeros(C.catq_ternary_infer_sync_bytes() // 4, dtype=torch.int32, device=device)
    outs = []
    for _ in range(2):
        C.catq_ternary_infer_staged(layers, stages, g, sync)
        torch.cuda.synchronize()
        assert C.catq_device_status() == 0
        assert int(sync.abs().sum().item()) == 0
        outs.append([y.clone() for y in ys])
    for a, b in zip(*outs):
        assert torch.equal(a, b)
    for codes, alpha, N, K, X, Y, mu in layers:
        ref = O.ternary_infer(U.to_host(codes), U.to_host(alpha), N, K, g, U.to_host(X),
                              mu=U.to_host(mu) if mu is not None else None)
        got = U.to_host(Y)
        assert np.isfinite(got).all(), (N, K)
        assert U.fro_rel(got, ref) <= U.TOL_BF16, (N, K)


def test_ternary_infer_staged_many_stages(device):
    """The most stages a call takes, each a small layer reading the previous one's output."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    g, B, D = 64, 2, 256
    n = C.catq_ternary_infer_max_stages()
    x0 = U.to_device(syn.round_bf16(syn.rng(9, "infer_staged/many").standard_normal((B, D)).astype(np.float32)),
                     "bf16", device)
    layers, ys = [], []
    for s in range(n):
        codes, alpha, _ = _packed_layer(device, D, D, g, f"many/{s}")
        Y = torch.full((B, D), float("nan"), dtype=torch.bfloat16, device=device)
        layers.append((codes, alpha, D, D, x0 if s == 0 else ys[-1], Y, None))
        ys.append(Y)
    sync = torch.zeros(C.catq_ternary_infer_sync_bytes() // 4, dtype=torch.int32, device=device)
    C.catq_ternary_infer_staged(layers, list(range(n)), g, sync)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    assert int(sync.abs().sum().item()) == 0
    for codes, alpha, N, K, X, Y, _ in layers:
        ref = O.ternary_infer(U.to_host(codes), U.to_host(alpha), N, K, g, U.to_host(X))
        assert U.fro_rel(U.to_host(Y), ref) <= U.TOL_BF16


def test_ternary_infer_staged_rejects_bad_stages(device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    codes, alpha, _ = _packed_layer(device, 256, 256, 64, "bad")
    X = torch.zeros(1, 256, dtype=torch.bfloat16, device=device)
    Y = torch.zeros(1, 256, dtype=torch.bfloat16, device=device)
    Y2 = torch.zeros(1, 256, dtype=torch.bfloat16, device=device)
    sync = torch.zeros(C.catq_ternary_infer_sync_bytes() // 4, dtype=torch.int32, device=device)
    L = [(codes, alpha, 256, 256, X, Y, None), (codes, alpha, 256, 256, Y, Y2, None)]
    for bad in ([1, 1], [0, 2], [1, 0]):
        with pytest.raises(C.CatqError):
            C.catq_ternary_infer_staged(L, bad, 64, sync)
