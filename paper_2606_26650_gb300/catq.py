"""Python binding of libcatq (include/catq.h): argument marshalling only.

Every function here has the C name of the call it wraps, takes torch tensors that live on
the current CUDA device, passes their data pointers and the current torch stream to the
library, and raises CatqError on a non-zero status.  All arithmetic runs in the library's
CUDA kernels; there is no fallback.  PyTorch provides device memory and streams.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import re

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libcatq.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "catq.h")

F32, BF16 = 0, 1
PHASE_TEACHER, PHASE_SOFT, PHASE_HARD = 0, 1, 2
THR_HALF, THR_TWN07, THR_ABSMEAN, THR_TWN_STATIC = 0, 1, 2, 3
REDUCE_MEAN, REDUCE_SUM = 0, 1
RECON_ALPHA_T, RECON_ALPHA_T_MU = 0, 1

STATUS = {
    0: "CATQ_OK", 1: "CATQ_ERR_INVALID_ARG", 2: "CATQ_ERR_SHAPE", 3: "CATQ_ERR_DTYPE",
    4: "CATQ_ERR_ALIGN", 5: "CATQ_ERR_CUDA", 6: "CATQ_ERR_TIMEOUT", 7: "CATQ_ERR_NONFINITE",
    8: "CATQ_ERR_UNSUPPORTED", 9: "CATQ_ERR_WORKSPACE",
}


class CatqError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)}")


class catq_layer(ctypes.Structure):
    _fields_ = [
        ("N", ctypes.c_int64), ("K", ctypes.c_int64), ("g", ctypes.c_int32), ("w_dtype", ctypes.c_int32),
        ("W", ctypes.c_void_p),
        ("mu0", ctypes.c_void_p), ("alpha0", ctypes.c_void_p), ("delta0", ctypes.c_void_p),
        ("d_mu", ctypes.c_void_p), ("d_alpha", ctypes.c_void_p), ("d_delta", ctypes.c_void_p),
        ("op_const", ctypes.c_void_p), ("recon", ctypes.c_int32), ("reserved", ctypes.c_int32),
    ]


class catq_grouped_layer(ctypes.Structure):
    _fields_ = [
        ("E", ctypes.c_int32), ("g", ctypes.c_int32), ("N", ctypes.c_int64), ("K", ctypes.c_int64),
        ("w_dtype", ctypes.c_int32), ("recon", ctypes.c_int32), ("W", ctypes.c_void_p),
        ("mu0", ctypes.c_void_p), ("alpha0", ctypes.c_void_p), ("delta0", ctypes.c_void_p),
        ("d_mu", ctypes.c_void_p), ("d_alpha", ctypes.c_void_p), ("d_delta", ctypes.c_void_p),
        ("op_const", ctypes.c_void_p),
    ]


class catq_schedule(ctypes.Structure):
    _fields_ = [("phase", ctypes.c_int32), ("s", ctypes.c_float)]


class catq_infer_layer(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("alpha", ctypes.c_void_p), ("mu", ctypes.c_void_p),
                ("N", ctypes.c_int64), ("K", ctypes.c_int64), ("X", ctypes.c_void_p), ("Y", ctypes.c_void_p)]


class catq_adamw(ctypes.Structure):
    _fields_ = [("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float),
                ("weight_decay", ctypes.c_float), ("margin", ctypes.c_float)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (there is no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
    L = ctypes.CDLL(LIB_PATH)
    P, I64, I32, F, S = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float, ctypes.c_size_t
    LP = ctypes.POINTER(catq_layer)
    sig = {
        "catq_abi_version": (I32, []),
        "catq_status_string": (ctypes.c_char_p, [I32]),
        "catq_group_stats": (I32, [LP, I32, P]),
        "catq_modulate_ternarize": (I32, [LP, catq_schedule, P, P, P, P]),
        "catq_soft_ternary_linear_fwd": (I32, [LP, catq_schedule, P, I64, I32, P, P]),
        "catq_bwd_workspace_bytes": (S, [LP, I64]),
        "catq_soft_ternary_linear_bwd": (I32, [LP, catq_schedule, P, P, I64, I32, P, P, P, P, P, S, P]),
        "catq_recon_loss_workspace_bytes": (S, [I64]),
        "catq_recon_loss": (I32, [P, P, I64, I32, I32, P, P, P, S, P]),
        "catq_hard_ternarize_pack": (I32, [LP, P, P, P, P]),
        "catq_device_status": (I32, [P, ctypes.POINTER(I32)]),
        "catq_selftest_wait_timeout": (I32, [ctypes.c_uint64, P]),
        "catq_ternary_infer": (I32, [P, P, P, I64, I64, I32, P, I64, I32, P, P]),
        "catq_soft_ternary_linear_bwd_noalloc": (I32, [LP, catq_schedule, P, P, I64, I32, P, P, P, P, P]),
        "catq_bwd_noalloc_max_scratch_bytes": (S, []),
        "catq_grouped_soft_ternary_linear_fwd": (I32, [ctypes.POINTER(catq_grouped_layer), catq_schedule, P, P, I32, P,
                                                       P]),
        "catq_grouped_bwd_workspace_bytes": (S, [ctypes.POINTER(catq_grouped_layer), P]),
        "catq_schedule_at_epoch": (I32, [I32, I32, ctypes.c_double, ctypes.c_double, ctypes.POINTER(catq_schedule)]),
        "catq_linear_decay_lr": (I32, [ctypes.c_double, I64, I64, ctypes.POINTER(F)]),
        "catq_factor_adamw_step": (I32, [I64, P, P, P, P, P, P, P, ctypes.POINTER(catq_adamw), I64, F, P]),
        "catq_grouped_soft_ternary_linear_bwd": (I32, [ctypes.POINTER(catq_grouped_layer), catq_schedule, P, P, P, I32,
                                                       P, P, P, P, P, S, P]),
        "catq_soft_ternary_linear_fwd_ex": (I32, [LP, catq_schedule, P, I64, I32, P, P, I32, P]),
        "catq_fwd_loss_workspace_bytes": (S, [LP, I64]),
        "catq_soft_ternary_linear_fwd_loss": (I32, [LP, catq_schedule, P, I64, I32, P, P, I32, I32, P, P, P, P, S, P]),
        "catq_act_quant_a8": (I32, [P, I64, I64, I32, P, P, P, P]),
        "catq_direct_adamw_step": (I32, [I64, P, P, P, P, P, ctypes.POINTER(catq_adamw), I64, F, P]),
        "catq_ternary_infer_max_layers": (I32, []),
        "catq_ternary_infer_batched": (I32, [ctypes.POINTER(catq_infer_layer), I32, I32, I64, I32, P]),
        "catq_ternary_infer_max_stages": (I32, []),
        "catq_ternary_infer_sync_bytes": (S, []),
        "catq_ternary_infer_staged": (I32, [ctypes.POINTER(catq_infer_layer), I32, ctypes.POINTER(I32), I32, I64, I32,
                                            P, P]),
        "catq_group_recon_error": (I32, [LP, P, P]),
        "catq_grouped_fwd_loss_workspace_bytes": (S, [ctypes.POINTER(catq_grouped_layer), P]),
        "catq_rmsnorm_fwd": (I32, [P, I32, P, P, I64, I64, F, P, P, P, P]),
        "catq_rmsnorm_bwd": (I32, [P, I32, P, P, P, P, P, I64, I64, P, P]),
        "catq_rope": (I32, [P, I64, I64, I32, I32, F, I32, P]),
        "catq_swiglu_fwd": (I32, [P, P, I64, P, P]),
        "catq_swiglu_bwd": (I32, [P, P, P, I64, P, P, P]),
        "catq_block_output_loss": (I32, [P, P, I64, P, I32, P, P, P, P, S, P]),
        "catq_attention_fwd": (I32, [P, P, P, I32, I32, I32, I32, I32, P, P, P]),
        "catq_attention_bwd": (I32, [P, P, P, P, P, P, I32, I32, I32, I32, I32, P, P, P, P, P]),
        "catq_grouped_soft_ternary_linear_fwd_loss": (I32, [ctypes.POINTER(catq_grouped_layer), catq_schedule, P, P,
                                                            I32, P, I32, P, P, P, P, S, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def header_functions(path: str = HEADER):
    """Names of the functions include/catq.h declares."""
    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(catq_[a-z0-9_]+)\s*\(", text)))


# ------------------------------------------------------------------ marshalling helpers

def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _check(status: int, where: str):
    if status != 0:
        raise CatqError(status, where)


def _buf(t, name: str, nbytes: int, where: str):
    """The library reads and writes `nbytes` bytes at a tensor's address without seeing its
    size or device: refuse a host tensor or one too small before the call, so that a
    caller's mistake raises here instead of touching memory the tensor does not own.
    None passes (the call decides whether the argument is optional)."""
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{where}: {name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{where}: {name} must be contiguous")
    have = t.numel() * t.element_size()
    if have < nbytes:
        raise ValueError(f"{where}: {name} holds {have} bytes, the call needs {nbytes}")


@dataclasses.dataclass
class Layer:
    """One linear layer's device state: W [N, K], the per-group arrays ([G] fp32) and the
    operand-constant array the fused GEMMs read ([4 G] fp32, [5 G] with mu in the
    reconstruction).  `recon`: RECON_ALPHA_T (W ~ alpha T) or RECON_ALPHA_T_MU."""
    W: object
    g: int
    mu0: object
    alpha0: object
    delta0: object
    d_mu: object
    d_alpha: object
    d_delta: object
    op_const: object = None
    recon: int = RECON_ALPHA_T

    @classmethod
    def create(cls, W, g, d_mu=None, d_alpha=None, d_delta=None, recon=RECON_ALPHA_T):
        """Allocates the statistics, operand-constant and (identity, unless given) factor
        tensors."""
        import torch
        N, K = W.shape
        G = N * K // g
        kw = dict(device=W.device, dtype=torch.float32)
        return cls(W, g, torch.empty(G, **kw), torch.empty(G, **kw), torch.empty(G, **kw),
                   d_mu if d_mu is not None else torch.zeros(G, **kw),
                   d_alpha if d_alpha is not None else torch.ones(G, **kw),
                   d_delta if d_delta is not None else torch.ones(G, **kw),
                   torch.empty((5 if recon else 4) * G, **kw), int(recon))

    @property
    def N(self):
        return self.W.shape[0]

    @property
    def K(self):
        return self.W.shape[1]

    @property
    def G(self):
        return self.N * self.K // self.g

    def struct(self) -> catq_layer:
        G, where = self.G, "Layer"
        _buf(self.W, "W", self.N * self.K * self.W.element_size(), where)
        for name in ("mu0", "alpha0", "delta0", "d_mu", "d_alpha", "d_delta"):
            _buf(getattr(self, name), name, 4 * G, where)
        _buf(self.op_const, "op_const", 4 * (5 if self.recon else 4) * G, where)
        return catq_layer(self.N, self.K, self.g, _dtype_code(self.W), self.W.data_ptr(),
                          self.mu0.data_ptr(), self.alpha0.data_ptr(), self.delta0.data_ptr(),
                          self.d_mu.data_ptr(), self.d_alpha.data_ptr(), self.d_delta.data_ptr(),
                          self.op_const.data_ptr() if self.op_const is not None else None, self.recon, 0)


def schedule(phase: int, s: float = 0.0) -> catq_schedule:
    return catq_schedule(int(phase), float(s))


# ------------------------------------------------------------------ the C calls

def catq_group_stats(layer: Layer, thr_init: int = THR_HALF, stream=None):
    st = layer.struct()
    _check(lib().catq_group_stats(ctypes.byref(st), int(thr_init), _stream(stream)), "catq_group_stats")


def catq_modulate_ternarize(layer: Layer, sched: catq_schedule, Wq_out=None, T_out=None, alpha_out=None,
                            stream=None):
    st = layer.struct()
    w = "catq_modulate_ternarize"
    _buf(Wq_out, "Wq_out", layer.N * layer.K * layer.W.element_size(), w)
    _buf(T_out, "T_out", layer.N * layer.K, w)
    _buf(alpha_out, "alpha_out", 4 * layer.G, w)
    _check(lib().catq_modulate_ternarize(ctypes.byref(st), sched, _ptr(Wq_out), _ptr(T_out), _ptr(alpha_out),
                                         _stream(stream)), "catq_modulate_ternarize")


def catq_soft_ternary_linear_fwd(layer: Layer, sched: catq_schedule, X, Y, stream=None):
    st = layer.struct()
    M, e, w = X.shape[0], X.element_size(), "catq_soft_ternary_linear_fwd"
    _buf(X, "X", M * layer.K * e, w)
    _buf(Y, "Y", M * layer.N * e, w)
    _check(lib().catq_soft_ternary_linear_fwd(ctypes.byref(st), sched, _ptr(X), X.shape[0], _dtype_code(X),
                                              _ptr(Y), _stream(stream)), "catq_soft_ternary_linear_fwd")


def catq_soft_ternary_linear_fwd_ex(layer: Layer, sched: catq_schedule, X, Y, x_row_scale=None, stream=None):
    """Y = diag(x_row_scale) X Wq^T; Y may be fp32 for a bf16 layer."""
    st = layer.struct()
    M, w = X.shape[0], "catq_soft_ternary_linear_fwd_ex"
    _buf(X, "X", M * layer.K * X.element_size(), w)
    _buf(Y, "Y", M * layer.N * (Y.element_size() if Y is not None else 0), w)
    _buf(x_row_scale, "x_row_scale", 4 * M, w)
    _check(lib().catq_soft_ternary_linear_fwd_ex(ctypes.byref(st), sched, _ptr(X), M, _dtype_code(X),
                                                 _ptr(x_row_scale), _ptr(Y), _dtype_code(Y), _stream(stream)), w)


def catq_fwd_loss_workspace_bytes(layer: Layer, M: int) -> int:
    st = layer.struct()
    return int(lib().catq_fwd_loss_workspace_bytes(ctypes.byref(st), int(M)))


def catq_soft_ternary_linear_fwd_loss(layer: Layer, sched: catq_schedule, X, Y_ref, loss_out, dY, Y=None,
                                      x_row_scale=None, workspace=None, reduction: int = REDUCE_MEAN, stream=None):
    """Forward, Eq. 7 loss and dY in one pass; Y_ref may be fp32 for a bf16 layer."""
    st = layer.struct()
    M, e, w = X.shape[0], X.element_size(), "catq_soft_ternary_linear_fwd_loss"
    _buf(X, "X", M * layer.K * e, w)
    _buf(Y_ref, "Y_ref", M * layer.N * Y_ref.element_size(), w)
    _buf(dY, "dY", M * layer.N * e, w)
    _buf(Y, "Y", M * layer.N * e, w)
    _buf(loss_out, "loss_out", 4, w)
    _buf(x_row_scale, "x_row_scale", 4 * M, w)
    _buf(workspace, "workspace", 0, w)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().catq_soft_ternary_linear_fwd_loss(ctypes.byref(st), sched, _ptr(X), M, _dtype_code(X),
                                                   _ptr(x_row_scale), _ptr(Y_ref), _dtype_code(Y_ref),
                                                   int(reduction), _ptr(loss_out), _ptr(dY), _ptr(Y),
                                                   _ptr(workspace), ws_bytes, _stream(stream)), w)


def catq_act_quant_a8(X, codes, scale, X_deq=None, stream=None):
    """Per-token 8-bit codes (as exact values of X's dtype), scales [M] and (optionally) the
    dequantized activations."""
    M, K = X.shape
    n, w = M * K * X.element_size(), "catq_act_quant_a8"
    _buf(X, "X", n, w)
    _buf(codes, "codes", n, w)
    _buf(X_deq, "X_deq", n, w)
    _buf(scale, "scale", 4 * M, w)
    _check(lib().catq_act_quant_a8(_ptr(X), M, K, _dtype_code(X), _ptr(codes), _ptr(scale), _ptr(X_deq),
                                   _stream(stream)), w)


def catq_bwd_workspace_bytes(layer: Layer, M: int) -> int:
    st = layer.struct()
    return int(lib().catq_bwd_workspace_bytes(ctypes.byref(st), int(M)))


def catq_soft_ternary_linear_bwd(layer: Layer, sched: catq_schedule, X, dY, dX=None, g_dmu=None, g_dalpha=None,
                                 g_ddelta=None, workspace=None, stream=None):
    st = layer.struct()
    _bwd_bufs(layer, X, dY, dX, (g_dmu, g_dalpha, g_ddelta), "catq_soft_ternary_linear_bwd")
    _buf(workspace, "workspace", 0, "catq_soft_ternary_linear_bwd")
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().catq_soft_ternary_linear_bwd(ctypes.byref(st), sched, _ptr(X), _ptr(dY), X.shape[0],
                                              _dtype_code(X), _ptr(dX), _ptr(g_dmu), _ptr(g_dalpha),
                                              _ptr(g_ddelta), _ptr(workspace), ws_bytes, _stream(stream)),
           "catq_soft_ternary_linear_bwd")


def catq_soft_ternary_linear_bwd_noalloc(layer: Layer, sched: catq_schedule, X, dY, dX=None, g_dmu=None,
                                         g_dalpha=None, g_ddelta=None, stream=None):
    st = layer.struct()
    _bwd_bufs(layer, X, dY, dX, (g_dmu, g_dalpha, g_ddelta), "catq_soft_ternary_linear_bwd_noalloc")
    _check(lib().catq_soft_ternary_linear_bwd_noalloc(ctypes.byref(st), sched, _ptr(X), _ptr(dY), X.shape[0],
                                                      _dtype_code(X), _ptr(dX), _ptr(g_dmu), _ptr(g_dalpha),
                                                      _ptr(g_ddelta), _stream(stream)),
           "catq_soft_ternary_linear_bwd_noalloc")


def _bwd_bufs(layer, X, dY, dX, grads, where, rows=None, groups=None):
    M = X.shape[0] if rows is None else rows
    e = X.element_size()
    _buf(X, "X", M * layer.K * e, where)
    _buf(dY, "dY", M * layer.N * e, where)
    _buf(dX, "dX", M * layer.K * e, where)
    for name, arr in zip(("g_dmu", "g_dalpha", "g_ddelta"), grads):
        _buf(arr, name, 4 * (layer.G if groups is None else groups), where)


def catq_bwd_noalloc_max_scratch_bytes() -> int:
    return int(lib().catq_bwd_noalloc_max_scratch_bytes())


def catq_recon_loss_workspace_bytes(count: int) -> int:
    return int(lib().catq_recon_loss_workspace_bytes(int(count)))


def catq_recon_loss(Y, Y_ref, loss_out, dY=None, workspace=None, reduction: int = REDUCE_MEAN, stream=None):
    w, n = "catq_recon_loss", Y.numel() * Y.element_size()
    _buf(Y, "Y", n, w)
    _buf(Y_ref, "Y_ref", n, w)
    _buf(dY, "dY", n, w)
    _buf(loss_out, "loss_out", 4, w)
    _buf(workspace, "workspace", 0, w)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().catq_recon_loss(_ptr(Y), _ptr(Y_ref), Y.numel(), _dtype_code(Y), int(reduction), _ptr(loss_out),
                                 _ptr(dY), _ptr(workspace), ws_bytes, _stream(stream)), "catq_recon_loss")


def catq_hard_ternarize_pack(layer: Layer, codes, alpha=None, mu=None, stream=None):
    st = layer.struct()
    w = "catq_hard_ternarize_pack"
    _buf(codes, "codes", layer.N * layer.K // 4, w)
    _buf(alpha, "alpha", 4 * layer.G, w)
    _buf(mu, "mu", 4 * layer.G, w)
    _check(lib().catq_hard_ternarize_pack(ctypes.byref(st), _ptr(codes), _ptr(alpha), _ptr(mu), _stream(stream)),
           "catq_hard_ternarize_pack")


def catq_device_status(stream=None) -> int:
    out = ctypes.c_int32(0)
    _check(lib().catq_device_status(_stream(stream), ctypes.byref(out)), "catq_device_status")
    return int(out.value)


def catq_ternary_infer(codes, alpha, N: int, K: int, g: int, X, Y, mu=None, stream=None):
    """Y [B, N] = X [B, K] (alpha T + mu)^T from the 2-bit codes, group scales and (for the
    W ~ alpha T + mu form) group offsets of catq_hard_ternarize_pack."""
    w, B, G = "catq_ternary_infer", X.shape[0], int(N) * int(K) // max(int(g), 1)
    _buf(codes, "codes", int(N) * int(K) // 4, w)
    _buf(alpha, "alpha", 4 * G, w)
    _buf(mu, "mu", 4 * G, w)
    _buf(X, "X", B * int(K) * X.element_size(), w)
    _buf(Y, "Y", B * int(N) * X.element_size(), w)
    _check(lib().catq_ternary_infer(_ptr(codes), _ptr(alpha), _ptr(mu), int(N), int(K), int(g), _ptr(X),
                                    X.shape[0], _dtype_code(X), _ptr(Y), _stream(stream)), "catq_ternary_infer")


def catq_ternary_infer_max_layers() -> int:
    return int(lib().catq_ternary_infer_max_layers())


def catq_ternary_infer_batched(layers, g: int, stream=None):
    """Several independent layers in one launch: `layers` is a list of tuples
    (codes, alpha, N, K, X, Y, mu) (mu may be None), all with the same token rows X.shape[0]."""
    w = "catq_ternary_infer_batched"
    arr = (catq_infer_layer * max(1, len(layers)))()
    B = layers[0][4].shape[0] if layers else 0
    for i, (codes, alpha, N, K, X, Y, mu) in enumerate(layers):
        G = int(N) * int(K) // max(int(g), 1)
        _buf(codes, "codes", int(N) * int(K) // 4, w)
        _buf(alpha, "alpha", 4 * G, w)
        _buf(mu, "mu", 4 * G, w)
        if X.shape[0] != B:
            raise ValueError(f"{w}: every layer needs the same token rows ({B})")
        _buf(X, "X", B * int(K) * X.element_size(), w)
        _buf(Y, "Y", B * int(N) * X.element_size(), w)
        arr[i] = catq_infer_layer(codes.data_ptr(), alpha.data_ptr(), mu.data_ptr() if mu is not None else None,
                                  int(N), int(K), X.data_ptr(), Y.data_ptr())
    dt = _dtype_code(layers[0][4]) if layers else BF16
    _check(lib().catq_ternary_infer_batched(arr, len(layers), int(g), int(B), dt, _stream(stream)), w)


def _infer_layer_array(layers, g, w):
    arr = (catq_infer_layer * max(1, len(layers)))()
    B = layers[0][4].shape[0] if layers else 0
    for i, (codes, alpha, N, K, X, Y, mu) in enumerate(layers):
        G = int(N) * int(K) // max(int(g), 1)
        _buf(codes, "codes", int(N) * int(K) // 4, w)
        _buf(alpha, "alpha", 4 * G, w)
        _buf(mu, "mu", 4 * G, w)
        if X.shape[0] != B:
            raise ValueError(f"{w}: every layer needs the same token rows ({B})")
        _buf(X, "X", B * int(K) * X.element_size(), w)
        _buf(Y, "Y", B * int(N) * X.element_size(), w)
        arr[i] = catq_infer_layer(codes.data_ptr(), alpha.data_ptr(), mu.data_ptr() if mu is not None else None,
                                  int(N), int(K), X.data_ptr(), Y.data_ptr())
    return arr, B


def catq_ternary_infer_sync_bytes() -> int:
    return int(lib().catq_ternary_infer_sync_bytes())


def catq_ternary_infer_max_stages() -> int:
    return int(lib().catq_ternary_infer_max_stages())


def catq_ternary_infer_staged(layers, stages, g: int, sync, stream=None):
    """Layers in dependency order in one cooperative launch: `layers` as in
    catq_ternary_infer_batched, `stages` the stage of each layer (0, then non-decreasing in steps
    of 1); a layer may read the Y of a layer of an earlier stage.  `sync`: a zeroed device buffer
    of catq_ternary_infer_sync_bytes() bytes (left zeroed)."""
    w = "catq_ternary_infer_staged"
    arr, B = _infer_layer_array(layers, g, w)
    _buf(sync, "sync", catq_ternary_infer_sync_bytes(), w)
    st = (ctypes.c_int32 * max(1, len(stages)))(*[int(v) for v in stages])
    if len(stages) != len(layers):
        raise ValueError(f"{w}: one stage per layer")
    dt = _dtype_code(layers[0][4]) if layers else BF16
    _check(lib().catq_ternary_infer_staged(arr, len(layers), st, int(g), int(B), dt, _ptr(sync), _stream(stream)), w)


def catq_schedule_at_epoch(e: int, m: int = 60, gamma: float = 0.8, s0: float = 30.0) -> catq_schedule:
    """Eq. 6's (phase, s) of calibration epoch e of m (host only)."""
    out = catq_schedule()
    _check(lib().catq_schedule_at_epoch(int(e), int(m), float(gamma), float(s0), ctypes.byref(out)),
           "catq_schedule_at_epoch")
    return out


def catq_linear_decay_lr(lr0: float, k: int, total: int) -> float:
    """Learning rate of update k of `total` under a linear decay to zero (host only)."""
    out = ctypes.c_float()
    _check(lib().catq_linear_decay_lr(float(lr0), int(k), int(total), ctypes.byref(out)), "catq_linear_decay_lr")
    return float(out.value)


def adamw(beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8, weight_decay: float = 0.0,
          margin: float = 1e-4) -> catq_adamw:
    return catq_adamw(beta1, beta2, eps, weight_decay, margin)


def catq_factor_adamw_step(d_mu, d_alpha, d_delta, g_dmu, g_dalpha, g_ddelta, moments, hp: catq_adamw, t: int,
                           lr: float, stream=None):
    """One AdamW update of the factors [G] in place from their gradients; moments [6 * G]
    (zero before the first update) is the optimizer state."""
    G, w = d_mu.numel(), "catq_factor_adamw_step"
    for name, arr in zip(("d_mu", "d_alpha", "d_delta", "g_dmu", "g_dalpha", "g_ddelta"),
                         (d_mu, d_alpha, d_delta, g_dmu, g_dalpha, g_ddelta)):
        _buf(arr, name, 4 * G, w)
    _buf(moments, "moments", 4 * 6 * G, w)
    _check(lib().catq_factor_adamw_step(d_mu.numel(), _ptr(d_mu), _ptr(d_alpha), _ptr(d_delta), _ptr(g_dmu),
                                        _ptr(g_dalpha), _ptr(g_ddelta), _ptr(moments), ctypes.byref(hp), int(t),
                                        float(lr), _stream(stream)), "catq_factor_adamw_step")


def catq_direct_adamw_step(d_alpha, d_delta, g_dalpha, g_ddelta, moments, hp: catq_adamw, t: int, lr: float,
                           stream=None):
    """Direct learning's update of (d_alpha, d_delta) [G] in place; moments [4 * G]."""
    G, w = d_alpha.numel(), "catq_direct_adamw_step"
    for name, arr in zip(("d_alpha", "d_delta", "g_dalpha", "g_ddelta"), (d_alpha, d_delta, g_dalpha, g_ddelta)):
        _buf(arr, name, 4 * G, w)
    _buf(moments, "moments", 4 * 4 * G, w)
    _check(lib().catq_direct_adamw_step(G, _ptr(d_alpha), _ptr(d_delta), _ptr(g_dalpha), _ptr(g_ddelta),
                                        _ptr(moments), ctypes.byref(hp), int(t), float(lr), _stream(stream)), w)


def catq_group_recon_error(layer: Layer, err, stream=None):
    """err [G] = per-group mean of (W - Wq)^2 for the hard reconstruction."""
    st = layer.struct()
    _buf(err, "err", 4 * layer.G, "catq_group_recon_error")
    _check(lib().catq_group_recon_error(ctypes.byref(st), _ptr(err), _stream(stream)), "catq_group_recon_error")


def catq_selftest_wait_timeout(timeout_ns: int, stream=None):
    _check(lib().catq_selftest_wait_timeout(int(timeout_ns), _stream(stream)), "catq_selftest_wait_timeout")


def workspace(nbytes: int, device):
    """A byte tensor of at least nbytes (256-byte aligned by the caching allocator)."""
    import torch
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# ------------------------------------------------------------------ grouped (MoE) layers

@dataclasses.dataclass
class GroupedLayer:
    """E experts stacked: W [E, N, K], per-group arrays [E * G] (expert-major).  `dense`
    views the stack as one [E * N, K] layer for catq_group_stats / pack."""
    W: object
    g: int
    dense: Layer

    @classmethod
    def create(cls, W, g, d_mu=None, d_alpha=None, d_delta=None, recon=RECON_ALPHA_T):
        E, N, K = W.shape
        return cls(W, g, Layer.create(W.reshape(E * N, K), g, d_mu, d_alpha, d_delta, recon))

    @property
    def E(self):
        return self.W.shape[0]

    def struct(self) -> catq_grouped_layer:
        E, N, K = self.W.shape
        d = self.dense
        d.struct()  # checks the stacked weights and the [E * G] per-group arrays
        return catq_grouped_layer(E, self.g, N, K, _dtype_code(self.W), d.recon, self.W.data_ptr(), d.mu0.data_ptr(),
                                  d.alpha0.data_ptr(), d.delta0.data_ptr(), d.d_mu.data_ptr(), d.d_alpha.data_ptr(),
                                  d.d_delta.data_ptr(), d.op_const.data_ptr() if d.op_const is not None else None)


def _offsets(row_offsets):
    arr = (ctypes.c_int64 * len(row_offsets))(*[int(v) for v in row_offsets])
    return arr


def _grouped_bufs(layer, row_offsets, where, X=None, Y=None, dY=None, dX=None, grads=()):
    """The library reads E + 1 row offsets and rows 0 .. R-1 of the row-indexed arrays."""
    E, N, K = layer.W.shape
    if len(row_offsets) != E + 1:
        raise ValueError(f"{where}: row_offsets has {len(row_offsets)} entries, the layer's {E} experts need {E + 1}")
    R = int(row_offsets[-1])
    e = X.element_size() if X is not None else 2
    _buf(X, "X", R * K * e, where)
    _buf(Y, "Y", R * N * e, where)
    _buf(dY, "dY", R * N * e, where)
    _buf(dX, "dX", R * K * e, where)
    for name, arr in zip(("g_dmu", "g_dalpha", "g_ddelta"), grads):
        _buf(arr, name, 4 * E * (N * K // layer.g), where)


def catq_grouped_soft_ternary_linear_fwd(layer: GroupedLayer, sched: catq_schedule, X, row_offsets, Y, stream=None):
    st = layer.struct()
    _grouped_bufs(layer, row_offsets, "catq_grouped_soft_ternary_linear_fwd", X=X, Y=Y)
    off = _offsets(row_offsets)
    _check(lib().catq_grouped_soft_ternary_linear_fwd(ctypes.byref(st), sched, _ptr(X), off, _dtype_code(X), _ptr(Y),
                                                      _stream(stream)), "catq_grouped_soft_ternary_linear_fwd")


def catq_grouped_bwd_workspace_bytes(layer: GroupedLayer, row_offsets) -> int:
    st = layer.struct()
    _grouped_bufs(layer, row_offsets, "catq_grouped_bwd_workspace_bytes")
    return int(lib().catq_grouped_bwd_workspace_bytes(ctypes.byref(st), _offsets(row_offsets)))


def catq_grouped_soft_ternary_linear_bwd(layer: GroupedLayer, sched: catq_schedule, X, dY, row_offsets, dX=None,
                                         g_dmu=None, g_dalpha=None, g_ddelta=None, workspace=None, stream=None):
    st = layer.struct()
    _grouped_bufs(layer, row_offsets, "catq_grouped_soft_ternary_linear_bwd", X=X, dY=dY, dX=dX,
                  grads=(g_dmu, g_dalpha, g_ddelta))
    _buf(workspace, "workspace", 0, "catq_grouped_soft_ternary_linear_bwd")
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().catq_grouped_soft_ternary_linear_bwd(ctypes.byref(st), sched, _ptr(X), _ptr(dY),
                                                      _offsets(row_offsets), _dtype_code(X), _ptr(dX), _ptr(g_dmu),
                                                      _ptr(g_dalpha), _ptr(g_ddelta), _ptr(workspace), ws_bytes,
                                                      _stream(stream)), "catq_grouped_soft_ternary_linear_bwd")


def catq_grouped_fwd_loss_workspace_bytes(layer: GroupedLayer, row_offsets) -> int:
    st = layer.struct()
    _grouped_bufs(layer, row_offsets, "catq_grouped_fwd_loss_workspace_bytes")
    return int(lib().catq_grouped_fwd_loss_workspace_bytes(ctypes.byref(st), _offsets(row_offsets)))


def catq_grouped_soft_ternary_linear_fwd_loss(layer: GroupedLayer, sched: catq_schedule, X, row_offsets, Y_ref,
                                              loss_out, dY, Y=None, workspace=None, reduction: int = REDUCE_MEAN,
                                              stream=None):
    st = layer.struct()
    w = "catq_grouped_soft_ternary_linear_fwd_loss"
    _grouped_bufs(layer, row_offsets, w, X=X, Y=Y, dY=dY)
    _grouped_bufs(layer, row_offsets, w, Y=Y_ref)
    _buf(loss_out, "loss_out", 4, w)
    _buf(workspace, "workspace", 0, w)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().catq_grouped_soft_ternary_linear_fwd_loss(ctypes.byref(st), sched, _ptr(X), _offsets(row_offsets),
                                                           _dtype_code(X), _ptr(Y_ref), int(reduction),
                                                           _ptr(loss_out), _ptr(dY), _ptr(Y), _ptr(workspace),
                                                           ws_bytes, _stream(stream)), w)


# ------------------------------------------------------------------ decoder-block layers
# bf16 activations [T, *] (tokens t = b S + s); fp32 gamma, r, lse, delta.

def _bf16_bufs(where, nbytes, **bufs):
    import torch
    for name, t in bufs.items():
        if t is not None and t.dtype != torch.bfloat16:
            raise ValueError(f"{where}: {name} must be bfloat16")
        _buf(t, name, nbytes, where)


def catq_rmsnorm_fwd(X, gamma, Z, r, eps, residual=None, h_out=None, stream=None):
    """Z = gamma * h / rms(h), h = X (+ residual, in fp32, stored into h_out); r [T] = 1 / rms(h).
    X bf16 or fp32; residual, Z bf16; h_out fp32."""
    import torch
    T, H = X.shape
    w = "catq_rmsnorm_fwd"
    _buf(X, "X", T * H * X.element_size(), w)
    _bf16_bufs(w, 2 * T * H, residual=residual, Z=Z)
    if h_out is not None and h_out.dtype != torch.float32:
        raise ValueError(f"{w}: h_out must be float32")
    _buf(h_out, "h_out", 4 * T * H, w)
    _buf(gamma, "gamma", 4 * H, w)
    _buf(r, "r", 4 * T, w)
    _check(lib().catq_rmsnorm_fwd(_ptr(X), _dtype_code(X), _ptr(residual), _ptr(gamma), T, H, float(eps),
                                  _ptr(h_out), _ptr(Z), _ptr(r), _stream(stream)), w)


def catq_rmsnorm_bwd(h, gamma, r, dZ, dX, dZ2=None, d_residual=None, stream=None):
    """dX of catq_rmsnorm_fwd at h (bf16 or fp32); dZ, dZ2, d_residual, dX bf16."""
    T, H = h.shape
    w = "catq_rmsnorm_bwd"
    _buf(h, "h", T * H * h.element_size(), w)
    _bf16_bufs(w, 2 * T * H, dZ=dZ, dZ2=dZ2, d_residual=d_residual, dX=dX)
    _buf(gamma, "gamma", 4 * H, w)
    _buf(r, "r", 4 * T, w)
    _check(lib().catq_rmsnorm_bwd(_ptr(h), _dtype_code(h), _ptr(gamma), _ptr(r), _ptr(dZ), _ptr(dZ2),
                                  _ptr(d_residual), T, H, _ptr(dX), _stream(stream)), w)


def catq_rope(X, S, n_heads, d, base, inverse=False, stream=None):
    T = X.shape[0]
    w = "catq_rope"
    _bf16_bufs(w, 2 * T * n_heads * d, X=X)
    _check(lib().catq_rope(_ptr(X), T, int(S), int(n_heads), int(d), float(base), int(bool(inverse)),
                           _stream(stream)), w)


def catq_swiglu_fwd(gate, up, M, stream=None):
    n = gate.numel()
    _bf16_bufs("catq_swiglu_fwd", 2 * n, gate=gate, up=up, M=M)
    _check(lib().catq_swiglu_fwd(_ptr(gate), _ptr(up), n, _ptr(M), _stream(stream)), "catq_swiglu_fwd")


def catq_swiglu_bwd(gate, up, dM, d_gate, d_up, stream=None):
    n = gate.numel()
    _bf16_bufs("catq_swiglu_bwd", 2 * n, gate=gate, up=up, dM=dM, d_gate=d_gate, d_up=d_up)
    _check(lib().catq_swiglu_bwd(_ptr(gate), _ptr(up), _ptr(dM), n, _ptr(d_gate), _ptr(d_up), _stream(stream)),
           "catq_swiglu_bwd")


def catq_block_output_loss(h, branch, out_ref=None, loss_out=None, d_out=None, out=None, workspace=None,
                           reduction: int = REDUCE_MEAN, stream=None):
    """out = h + branch in fp32; with out_ref, Eq. 7's loss into loss_out and d_out (bf16)."""
    import torch
    n, w = h.numel(), "catq_block_output_loss"
    for name, t in (("h", h), ("out_ref", out_ref), ("out", out)):
        if t is not None and t.dtype != torch.float32:
            raise ValueError(f"{w}: {name} must be float32")
        _buf(t, name, 4 * n, w)
    _bf16_bufs(w, 2 * n, branch=branch, d_out=d_out)
    _buf(loss_out, "loss_out", 4, w)
    _buf(workspace, "workspace", 0, w)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib().catq_block_output_loss(_ptr(h), _ptr(branch), n, _ptr(out_ref), int(reduction), _ptr(loss_out),
                                        _ptr(d_out), _ptr(out), _ptr(workspace), ws_bytes, _stream(stream)), w)


def catq_attention_fwd(Q, K, V, O, lse, B, S, n_heads, n_kv_heads, d, stream=None):
    w = "catq_attention_fwd"
    _bf16_bufs(w, 2 * B * S * n_heads * d, Q=Q, O=O)
    _bf16_bufs(w, 2 * B * S * n_kv_heads * d, K=K, V=V)
    _buf(lse, "lse", 4 * B * n_heads * S, w)
    _check(lib().catq_attention_fwd(_ptr(Q), _ptr(K), _ptr(V), int(B), int(S), int(n_heads), int(n_kv_heads),
                                    int(d), _ptr(O), _ptr(lse), _stream(stream)), w)


def catq_attention_bwd(Q, K, V, O, dO, lse, delta, dQ, dK, dV, B, S, n_heads, n_kv_heads, d, stream=None):
    w = "catq_attention_bwd"
    _bf16_bufs(w, 2 * B * S * n_heads * d, Q=Q, O=O, dO=dO, dQ=dQ)
    _bf16_bufs(w, 2 * B * S * n_kv_heads * d, K=K, V=V, dK=dK, dV=dV)
    _buf(lse, "lse", 4 * B * n_heads * S, w)
    _buf(delta, "delta", 4 * B * n_heads * S, w)
    _check(lib().catq_attention_bwd(_ptr(Q), _ptr(K), _ptr(V), _ptr(O), _ptr(dO), _ptr(lse), int(B), int(S),
                                    int(n_heads), int(n_kv_heads), int(d), _ptr(delta), _ptr(dQ), _ptr(dK),
                                    _ptr(dV), _stream(stream)), w)
