"""One decoder block as the window of Eq. 7's reconstruction (§2.4, a sliding window of one
block): the teacher block with full-precision weights, the student block whose seven linears
are soft-ternary (Eq. 6 weight at the schedule's point), the block-output loss, and every
linear's factor gradients through the block's backward.

Llama-family block (pre-norm, causal grouped-query attention with rotary position embedding,
SwiGLU MLP; with q_norm / k_norm the Qwen3 block, which normalises every query and key head);
tokens are rows t = b S + s of [B S, H] activations.  The linears' inputs and outputs are bf16; the residual stream (h = x + attention branch, out = h + MLP branch) stays in
fp32 and the loss is taken on the fp32 block output, so that the difference between student
and teacher is not lost to the rounding of a value the size of the residual.  The block input
x (bf16 or fp32) is the window's input and receives no gradient.  Every step here is a call
into libcatq (the linears, RMSNorm, rotary embedding, attention, SwiGLU, the block output and
its loss); this module only holds the buffers and orders the calls on one stream.
"""
from __future__ import annotations

import dataclasses

from . import catq as C

LINEARS = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


@dataclasses.dataclass(frozen=True)
class BlockShape:
    H: int          # hidden size
    n_heads: int
    n_kv_heads: int
    d: int          # head dimension
    I: int          # MLP intermediate size
    B: int          # sequences
    S: int          # tokens per sequence
    base: float = 500000.0
    eps: float = 1e-5

    @property
    def T(self):
        return self.B * self.S

    def linear_shapes(self):
        """(N, K) of each linear."""
        qd, kvd = self.n_heads * self.d, self.n_kv_heads * self.d
        return {"q_proj": (qd, self.H), "k_proj": (kvd, self.H), "v_proj": (kvd, self.H), "o_proj": (self.H, qd),
                "gate_proj": (self.I, self.H), "up_proj": (self.I, self.H), "down_proj": (self.H, self.I)}

    def linear_flops(self):
        """fwd + dX + dW of every linear: 6 T N K."""
        return float(sum(6.0 * self.T * n * k for n, k in self.linear_shapes().values()))

    def attention_flops(self):
        """Causal attention, forward (Q K^T and P V over the lower triangle: 2 B h S^2 d) and
        backward (five products: 5 B h S^2 d)."""
        return 7.0 * self.B * self.n_heads * self.S * self.S * self.d


class Block:
    """Device state and buffers of one block.  W: dict of bf16 [N, K] CUDA tensors by linear
    name; gamma1, gamma2: fp32 [H] norm weights; g: group size; factors: optional dict of
    (d_mu, d_alpha, d_delta) fp32 tensors by name (identity otherwise); q_norm, k_norm:
    optional fp32 [d] weights of the Qwen3 block's RMSNorm of every query and key head (applied
    to the projections' outputs before the rotary embedding)."""

    def __init__(self, shape: BlockShape, W, gamma1, gamma2, g, factors=None, thr_init=C.THR_HALF, stream=None,
                 q_norm=None, k_norm=None):
        import torch
        self.shape, self.g, self.stream = shape, g, stream
        dev = W["q_proj"].device
        self.device = dev
        for name, (n, k) in shape.linear_shapes().items():
            if tuple(W[name].shape) != (n, k) or W[name].dtype != torch.bfloat16:
                raise ValueError(f"{name}: expected bf16 [{n}, {k}], got {W[name].dtype} {tuple(W[name].shape)}")
        self.layers = {}
        for name in LINEARS:
            f = factors.get(name) if factors else None
            self.layers[name] = C.Layer.create(W[name], g, *(f if f is not None else (None, None, None)))
            C.catq_group_stats(self.layers[name], thr_init, stream=stream)
        self.gamma1, self.gamma2 = gamma1, gamma2
        if (q_norm is None) != (k_norm is None):
            raise ValueError("q_norm and k_norm come together")
        self.q_norm, self.k_norm = q_norm, k_norm
        T, H, I = shape.T, shape.H, shape.I
        qd, kvd = shape.n_heads * shape.d, shape.n_kv_heads * shape.d
        bf = dict(dtype=torch.bfloat16, device=dev)
        f32 = dict(dtype=torch.float32, device=dev)
        e = torch.empty
        # forward cache
        self.z1, self.r1 = e(T, H, **bf), e(T, **f32)
        self.q, self.k, self.v = e(T, qd, **bf), e(T, kvd, **bf), e(T, kvd, **bf)
        self.a, self.lse = e(T, qd, **bf), e(shape.B * shape.n_heads * shape.S, **f32)
        self.ao, self.h = e(T, H, **bf), e(T, H, **f32)
        self.z2, self.r2 = e(T, H, **bf), e(T, **f32)
        self.gt, self.u, self.m = e(T, I, **bf), e(T, I, **bf), e(T, I, **bf)
        self.dn = e(T, H, **bf)
        # backward
        self.d_out = e(T, H, **bf)
        self.dm, self.dgt, self.du = e(T, I, **bf), e(T, I, **bf), e(T, I, **bf)
        self.dz2a, self.dz2b, self.dh = e(T, H, **bf), e(T, H, **bf), e(T, H, **bf)
        self.da, self.dq, self.dk, self.dv = e(T, qd, **bf), e(T, qd, **bf), e(T, kvd, **bf), e(T, kvd, **bf)
        self.delta = e(shape.B * shape.n_heads * shape.S, **f32)
        if q_norm is not None:  # the projections' outputs before the head norm, and its RMS factors
            self.qp, self.kp = e(T, qd, **bf), e(T, kvd, **bf)
            self.rq, self.rk = e(T * shape.n_heads, **f32), e(T * shape.n_kv_heads, **f32)
        ws = max(C.catq_bwd_workspace_bytes(L, T) for L in self.layers.values())
        self.bwd_ws = C.workspace(ws, dev)
        self.loss_ws = C.workspace(C.catq_recon_loss_workspace_bytes(T * H), dev)

    # ---------------------------------------------------------------- forward
    def forward(self, x, sched, out=None, out_ref=None, loss=None, reduction=C.REDUCE_MEAN):
        """The block at schedule point sched (PHASE_TEACHER: full-precision weights), filling
        the forward cache the backward reads.  out: fp32 [T, H] block output (nullable);
        with out_ref, Eq. 7's loss into loss[0] and its gradient into the backward's d_out."""
        sh, st, L = self.shape, self.stream, self.layers
        C.catq_rmsnorm_fwd(x, self.gamma1, self.z1, self.r1, sh.eps, stream=st)
        if self.q_norm is None:
            C.catq_soft_ternary_linear_fwd(L["q_proj"], sched, self.z1, self.q, stream=st)
            C.catq_soft_ternary_linear_fwd(L["k_proj"], sched, self.z1, self.k, stream=st)
        else:
            C.catq_soft_ternary_linear_fwd(L["q_proj"], sched, self.z1, self.qp, stream=st)
            C.catq_soft_ternary_linear_fwd(L["k_proj"], sched, self.z1, self.kp, stream=st)
            C.catq_rmsnorm_fwd(self.qp.view(-1, sh.d), self.q_norm, self.q.view(-1, sh.d), self.rq, sh.eps, stream=st)
            C.catq_rmsnorm_fwd(self.kp.view(-1, sh.d), self.k_norm, self.k.view(-1, sh.d), self.rk, sh.eps, stream=st)
        C.catq_soft_ternary_linear_fwd(L["v_proj"], sched, self.z1, self.v, stream=st)
        C.catq_rope(self.q, sh.S, sh.n_heads, sh.d, sh.base, stream=st)
        C.catq_rope(self.k, sh.S, sh.n_kv_heads, sh.d, sh.base, stream=st)
        C.catq_attention_fwd(self.q, self.k, self.v, self.a, self.lse, sh.B, sh.S, sh.n_heads, sh.n_kv_heads, sh.d,
                             stream=st)
        C.catq_soft_ternary_linear_fwd(L["o_proj"], sched, self.a, self.ao, stream=st)
        C.catq_rmsnorm_fwd(x, self.gamma2, self.z2, self.r2, sh.eps, residual=self.ao, h_out=self.h, stream=st)
        C.catq_soft_ternary_linear_fwd(L["gate_proj"], sched, self.z2, self.gt, stream=st)
        C.catq_soft_ternary_linear_fwd(L["up_proj"], sched, self.z2, self.u, stream=st)
        C.catq_swiglu_fwd(self.gt, self.u, self.m, stream=st)
        C.catq_soft_ternary_linear_fwd(L["down_proj"], sched, self.m, self.dn, stream=st)
        C.catq_block_output_loss(self.h, self.dn, out_ref, loss, self.d_out if out_ref is not None else None, out,
                                 self.loss_ws, reduction=reduction, stream=st)

    # ---------------------------------------------------------------- one calibration step
    def teacher(self, x, out_ref):
        """out_ref (fp32 [T, H]) = the teacher block (full-precision weights) on x."""
        self.forward(x, C.schedule(C.PHASE_TEACHER), out=out_ref)

    def step(self, x, out_ref, sched, loss, grads, out=None, reduction=C.REDUCE_MEAN):
        """Forward at sched, loss[0] = Eq. 7's loss of the block output against out_ref (fp32),
        and grads[name] = (g_dmu, g_dalpha, g_ddelta) ([G] fp32 each, overwritten) of every
        linear.  out: fp32 [T, H] for the student output (not stored when None)."""
        sh, st, L = self.shape, self.stream, self.layers
        self.forward(x, sched, out=out, out_ref=out_ref, loss=loss, reduction=reduction)
        self._bwd("down_proj", sched, self.m, self.d_out, self.dm, grads)
        C.catq_swiglu_bwd(self.gt, self.u, self.dm, self.dgt, self.du, stream=st)
        self._bwd("gate_proj", sched, self.z2, self.dgt, self.dz2a, grads)
        self._bwd("up_proj", sched, self.z2, self.du, self.dz2b, grads)
        C.catq_rmsnorm_bwd(self.h, self.gamma2, self.r2, self.dz2a, self.dh, dZ2=self.dz2b, d_residual=self.d_out,
                           stream=st)
        self._bwd("o_proj", sched, self.a, self.dh, self.da, grads)
        C.catq_attention_bwd(self.q, self.k, self.v, self.a, self.da, self.lse, self.delta, self.dq, self.dk, self.dv,
                             sh.B, sh.S, sh.n_heads, sh.n_kv_heads, sh.d, stream=st)
        C.catq_rope(self.dq, sh.S, sh.n_heads, sh.d, sh.base, inverse=True, stream=st)
        C.catq_rope(self.dk, sh.S, sh.n_kv_heads, sh.d, sh.base, inverse=True, stream=st)
        if self.q_norm is not None:  # through the head norm, in place
            C.catq_rmsnorm_bwd(self.qp.view(-1, sh.d), self.q_norm, self.rq, self.dq.view(-1, sh.d),
                               self.dq.view(-1, sh.d), stream=st)
            C.catq_rmsnorm_bwd(self.kp.view(-1, sh.d), self.k_norm, self.rk, self.dk.view(-1, sh.d),
                               self.dk.view(-1, sh.d), stream=st)
        self._bwd("q_proj", sched, self.z1, self.dq, None, grads)
        self._bwd("k_proj", sched, self.z1, self.dk, None, grads)
        self._bwd("v_proj", sched, self.z1, self.dv, None, grads)
        return out

    def _bwd(self, name, sched, X, dY, dX, grads):
        g = grads[name]
        C.catq_soft_ternary_linear_bwd(self.layers[name], sched, X, dY, dX, g[0], g[1], g[2], workspace=self.bwd_ws,
                                       stream=self.stream)
