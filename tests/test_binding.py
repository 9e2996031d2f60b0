"""The Python binding's own checks, on the CPU: every buffer the library will read or write
must be a contiguous CUDA tensor of at least the size the call implies, and the grouped
calls need one row offset per expert plus one.  Mistakes raise ValueError before the
library is called, so none of them reaches a device."""
import numpy as np
import pytest

from paper_2606_26650_gb300 import catq as C

torch = pytest.importorskip("torch")


class FakeDev:
    """Stands in for a contiguous CUDA tensor: the checks read only these attributes."""

    def __init__(self, numel, elsize=4, cuda=True, contiguous=True, shape=None):
        self._n, self._e, self.is_cuda, self._c = numel, elsize, cuda, contiguous
        self.shape = shape if shape is not None else (numel,)
        self.dtype = {1: torch.uint8, 2: torch.bfloat16, 4: torch.float32}[elsize]

    def numel(self):
        return self._n

    def element_size(self):
        return self._e

    def is_contiguous(self):
        return self._c

    def data_ptr(self):
        return 4096


def test_buf_rules():
    C._buf(None, "x", 100, "t")                       # optional argument left out
    C._buf(FakeDev(25, 4), "x", 100, "t")             # exactly large enough
    with pytest.raises(ValueError, match="needs 100"):
        C._buf(FakeDev(24, 4), "x", 100, "t")
    with pytest.raises(ValueError, match="CUDA tensor"):
        C._buf(FakeDev(100, cuda=False), "x", 4, "t")
    with pytest.raises(ValueError, match="contiguous"):
        C._buf(FakeDev(100, contiguous=False), "x", 4, "t")


def _layer(N=64, K=256, g=128, short=None):
    G = N * K // g
    arrays = {n: FakeDev(G) for n in ("mu0", "alpha0", "delta0", "d_mu", "d_alpha", "d_delta")}
    if short:
        arrays[short] = FakeDev(G - 1)
    return C.Layer(FakeDev(N * K, 2, shape=(N, K)), g, op_const=FakeDev(4 * G), **arrays)


def test_layer_arrays_are_checked():
    assert _layer().struct().N == 64  # the layer itself is fine
    for name in ("mu0", "alpha0", "delta0", "d_mu", "d_alpha", "d_delta"):
        with pytest.raises(ValueError, match=name):
            _layer(short=name).struct()
    L = _layer()
    L.op_const = FakeDev(4 * L.G - 1)
    with pytest.raises(ValueError, match="op_const"):
        L.struct()


def test_host_tensors_are_refused_before_the_library():
    W = torch.zeros(64, 256, dtype=torch.bfloat16)
    layer = C.Layer.create(W, 128)  # CPU tensors throughout
    with pytest.raises(ValueError, match="CUDA tensor"):
        C.catq_group_stats(layer)


def test_call_sizes_follow_the_header():
    L = _layer()
    M, N, K = 10, L.N, L.K
    X, Y = FakeDev(M * K, 2, shape=(M, K)), FakeDev(M * N, 2, shape=(M, N))
    small_Y = FakeDev(M * N - 1, 2, shape=(M, N))
    with pytest.raises(ValueError, match="Y holds"):
        C.catq_soft_ternary_linear_fwd(L, C.schedule(C.PHASE_SOFT, 30.0), X, small_Y)
    with pytest.raises(ValueError, match="dX"):
        C._bwd_bufs(L, X, Y, FakeDev(M * K - 1, 2), (None, None, None), "bwd")
    with pytest.raises(ValueError, match="g_dalpha"):
        C._bwd_bufs(L, X, Y, None, (FakeDev(L.G), FakeDev(L.G - 1), FakeDev(L.G)), "bwd")
    with pytest.raises(ValueError, match="codes"):
        C.catq_hard_ternarize_pack(L, FakeDev(N * K // 4 - 1, 1))
    with pytest.raises(ValueError, match="dY"):
        C.catq_recon_loss(Y, Y, FakeDev(1), FakeDev(M * N - 1, 2))
    with pytest.raises(ValueError, match="alpha"):
        C.catq_ternary_infer(FakeDev(N * K // 4, 1), FakeDev(N * K // 128 - 1), N, K, 128,
                             FakeDev(K, 2, shape=(1, K)), FakeDev(N, 2, shape=(1, N)))
    with pytest.raises(ValueError, match="moments"):
        G = 10
        C.catq_factor_adamw_step(*(FakeDev(G) for _ in range(6)), FakeDev(6 * G - 1), C.adamw(), 1, 1e-3)


def test_grouped_offsets_and_rows():
    E, N, K, g = 3, 64, 256, 128
    G = N * K // g
    dense = C.Layer(FakeDev(E * N * K, 2, shape=(E * N, K)), g, *(FakeDev(E * G) for _ in range(6)),
                    op_const=FakeDev(4 * E * G))
    layer = C.GroupedLayer(FakeDev(E * N * K, 2, shape=(E, N, K)), g, dense)
    off = np.array([0, 4, 4, 9])
    X = FakeDev(9 * K, 2, shape=(9, K))
    C._grouped_bufs(layer, off, "t", X=X, Y=FakeDev(9 * N, 2))
    with pytest.raises(ValueError, match="row_offsets"):
        C._grouped_bufs(layer, off[:-1], "t", X=X)
    with pytest.raises(ValueError, match="Y holds"):
        C._grouped_bufs(layer, off, "t", X=X, Y=FakeDev(9 * N - 1, 2))
    with pytest.raises(ValueError, match="g_ddelta"):
        C._grouped_bufs(layer, off, "t", X=X, grads=(FakeDev(E * G), FakeDev(E * G), FakeDev(E * G - 1)))


def test_wrappers_pass_their_scalars_through(monkeypatch):
    """With valid buffers the wrappers reach the library with the caller's scalars (a fake
    library records the call)."""
    seen = {}

    class FakeLib:
        def __getattr__(self, name):
            def call(*args):
                seen[name] = args
                return 0
            return call

    monkeypatch.setattr(C, "lib", lambda: FakeLib())
    monkeypatch.setattr(C, "_stream", lambda stream=None: None)
    G = 10
    C.catq_factor_adamw_step(*(FakeDev(G) for _ in range(6)), FakeDev(6 * G), C.adamw(), 7, 5e-4)
    args = seen["catq_factor_adamw_step"]
    assert args[0] == G and args[-3] == 7 and args[-2] == pytest.approx(5e-4)
    L = _layer()
    M = 12
    X, Y = FakeDev(M * L.K, 2, shape=(M, L.K)), FakeDev(M * L.N, 2, shape=(M, L.N))
    C.catq_soft_ternary_linear_fwd(L, C.schedule(C.PHASE_SOFT, 30.0), X, Y)
    assert seen["catq_soft_ternary_linear_fwd"][3] == M
    C.catq_soft_ternary_linear_bwd(L, C.schedule(C.PHASE_SOFT, 30.0), X, Y, None,
                                   *(FakeDev(L.G) for _ in range(3)), workspace=FakeDev(256, 1))
    assert seen["catq_soft_ternary_linear_bwd"][4] == M
