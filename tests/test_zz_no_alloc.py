"""The allocation-free backward against the workspace backward, through the C ABI.

catq_soft_ternary_linear_bwd_noalloc serves callers that cannot allocate device memory:
it keeps the dW partial sums in a scratch array inside the library.  Its results must
equal those of catq_soft_ternary_linear_bwd (which uses a caller workspace) within the
tolerances of the other parity tests, call after call, since every call reuses the same
array.  This file sorts last so a stop-at-first-failure run has already run the rest.
"""
import ctypes

import numpy as np
import pytest

from paper_2606_26650_gb300 import catq as C
from paper_2606_26650_gb300 import synthetic as syn
from tests import gpu_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def device():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.device("cuda:0")


@pytest.mark.parametrize("dtype,N,K,g,M", [("bf16", 512, 384, 128, 700), ("f32", 192, 256, 64, 150)])
def test_noalloc_bwd_matches_workspace_bwd(device, dtype, N, K, g, M):
    import torch
    r = syn.rng(11, f"noalloc/{dtype}")
    W = r.standard_normal((N, K)).astype(np.float32) * 0.02
    X = r.standard_normal((M, K)).astype(np.float32)
    dY = r.standard_normal((M, N)).astype(np.float32) * 1e-3
    if dtype == "bf16":
        W, X, dY = syn.round_bf16(W), syn.round_bf16(X), syn.round_bf16(dY)
    G = N * K // g
    fac = [torch.from_numpy(f).to(device) for f in syn.factors(G, 11, f"noalloc/{dtype}", perturbed=True)]
    layer = C.Layer.create(U.to_device(W, dtype, device), g, *fac)
    C.catq_group_stats(layer)
    Xt, dYt = U.to_device(X, dtype, device), U.to_device(dY, dtype, device)
    sched = C.schedule(C.PHASE_SOFT, 15.0)

    ref_dX = torch.empty_like(Xt)
    ref = [torch.empty(G, device=device) for _ in range(3)]
    ws = C.workspace(C.catq_bwd_workspace_bytes(layer, M), device)
    C.catq_soft_ternary_linear_bwd(layer, sched, Xt, dYt, ref_dX, *ref, ws)
    torch.cuda.synchronize()
    for call in range(2):  # the second call reuses the scratch the first one left behind
        dX = torch.full_like(Xt, 3.0)
        got = [torch.full((G,), 5.0, device=device) for _ in range(3)]
        C.catq_soft_ternary_linear_bwd_noalloc(layer, sched, Xt, dYt, dX, *got)
        torch.cuda.synchronize()
        assert C.catq_device_status() == 0
        assert U.err(U.to_host(dX), U.to_host(ref_dX), dtype) <= U.tol(dtype), f"call {call}: dX"
        for a, b in zip(got, ref):
            assert U.err(U.to_host(a), U.to_host(b), dtype) <= U.tol(dtype), f"call {call}"


def test_noalloc_rejects_layers_beyond_its_scratch(device):
    """A layer whose partial sums exceed the scratch is refused before any launch."""
    lib = C.lib()
    limit = C.catq_bwd_noalloc_max_scratch_bytes()
    assert limit == 16 << 20
    N, K, g = 1 << 20, 64, 64  # 3 x N x (K / 64) x 4 bytes = 12 MiB per split ... scaled below
    while True:
        fake = C.catq_layer(N, K, g, C.F32, 16, 32, 64, 96, 128, 160, 192)
        if lib.catq_bwd_workspace_bytes(ctypes.byref(fake), 8) > limit:
            break
        N *= 2
    st = lib.catq_soft_ternary_linear_bwd_noalloc(ctypes.byref(fake), C.schedule(C.PHASE_SOFT, 30.0), 16, 16, 8,
                                                  C.F32, None, 256, 256, 256, None)
    assert st == 9  # CATQ_ERR_WORKSPACE
