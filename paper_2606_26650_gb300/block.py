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
its loss); this module only holds the buffers and orders the calls.

Calls that do not depend on each other run on side streams, joined by events: the q, k and v
projections (with their head norms and rotary embeddings) and the gate and up projections and
their dX contractions on a companion stream beside the main one, and every linear's
factor-gradient contraction (dW), which the backward's chain (dX, the layers between the
linears, attention) never waits for, in turn on the other side streams, each with its own dW
workspace.  A call of `forward` or `step` starts after the work already issued on the main
stream and ends with every side stream joined back into it.
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
                 q_norm=None, k_norm=None, side_streams=3):
        import torch
        self.shape, self.g, self.stream = shape, g, stream
        self.torch = torch
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
        # side streams (independent calls) and one dW workspace per side stream
        self.sides = [torch.cuda.Stream(device=dev) for _ in range(max(0, int(side_streams)))]
        self.bwd_ws = [C.workspace(ws, dev) for _ in range(1 + len(self.sides))]
        self.loss_ws = C.workspace(C.catq_recon_loss_workspace_bytes(T * H), dev)
        self._next_side = 0

    # ---------------------------------------------------------------- streams
    def _main(self):
        return self.stream if self.stream is not None else self.torch.cuda.current_stream(self.device)

    def _after(self, src, dst):
        """dst waits for the work issued so far on src."""
        if dst is not src:
            ev = self.torch.cuda.Event()
            ev.record(src)
            dst.wait_event(ev)

    def _side(self, i):
        """Side stream i (the main stream when the block has none)."""
        return self.sides[i % len(self.sides)] if self.sides else self._main()

    def _dw_lane(self, i):
        """The i-th dW stream and its workspace: the side streams after the companion (side 0),
        or side 0 itself when it is the only one, or the main stream."""
        lanes = list(range(1, len(self.sides))) or list(range(len(self.sides)))
        if not lanes:
            return self._main(), self.bwd_ws[0]
        j = lanes[i % len(lanes)]
        return self.sides[j], self.bwd_ws[1 + j]

    def _join(self):
        main = self._main()
        for sd in self.sides:
            self._after(sd, main)

    # ---------------------------------------------------------------- forward
    def forward(self, x, sched, out=None, out_ref=None, loss=None, reduction=C.REDUCE_MEAN):
        """The block at schedule point sched (PHASE_TEACHER: full-precision weights), filling
        the forward cache the backward reads.  out: fp32 [T, H] block output (nullable);
        with out_ref, Eq. 7's loss into loss[0] and its gradient into the backward's d_out."""
        self._forward(x, sched, out, out_ref, loss, reduction)
        self._join()

    def _forward(self, x, sched, out, out_ref, loss, reduction):
        sh, L = self.shape, self.layers
        st = self._main()
        sq, sk, sv = st, self._side(0), self._side(1)
        C.catq_rmsnorm_fwd(x, self.gamma1, self.z1, self.r1, sh.eps, stream=st)
        self._after(st, sk)
        self._after(st, sv)
        # q, k, v: each projection, head norm and rotary embedding on its own stream
        for name, y, yp, norm, r, nh, s_ in (("q_proj", self.q, "qp", self.q_norm, "rq", sh.n_heads, sq),
                                              ("k_proj", self.k, "kp", self.k_norm, "rk", sh.n_kv_heads, sk)):
            if norm is None:
                C.catq_soft_ternary_linear_fwd(L[name], sched, self.z1, y, stream=s_)
            else:
                pre = getattr(self, yp)
                C.catq_soft_ternary_linear_fwd(L[name], sched, self.z1, pre, stream=s_)
                C.catq_rmsnorm_fwd(pre.view(-1, sh.d), norm, y.view(-1, sh.d), getattr(self, r), sh.eps, stream=s_)
            C.catq_rope(y, sh.S, nh, sh.d, sh.base, stream=s_)
        C.catq_soft_ternary_linear_fwd(L["v_proj"], sched, self.z1, self.v, stream=sv)
        self._after(sk, st)
        self._after(sv, st)
        C.catq_attention_fwd(self.q, self.k, self.v, self.a, self.lse, sh.B, sh.S, sh.n_heads, sh.n_kv_heads, sh.d,
                             stream=st)
        C.catq_soft_ternary_linear_fwd(L["o_proj"], sched, self.a, self.ao, stream=st)
        C.catq_rmsnorm_fwd(x, self.gamma2, self.z2, self.r2, sh.eps, residual=self.ao, h_out=self.h, stream=st)
        su = self._side(0)
        self._after(st, su)
        C.catq_soft_ternary_linear_fwd(L["gate_proj"], sched, self.z2, self.gt, stream=st)
        C.catq_soft_ternary_linear_fwd(L["up_proj"], sched, self.z2, self.u, stream=su)
        self._after(su, st)
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
        sh, L = self.shape, self.layers
        st = self._main()
        self._next_side = 0
        self._forward(x, sched, out, out_ref, loss, reduction)
        self._dw("down_proj", sched, self.m, self.d_out, grads)
        self._dx("down_proj", sched, self.m, self.d_out, self.dm, st)
        C.catq_swiglu_bwd(self.gt, self.u, self.dm, self.dgt, self.du, stream=st)
        self._dw("gate_proj", sched, self.z2, self.dgt, grads)
        self._dw("up_proj", sched, self.z2, self.du, grads)
        su = self._side(0)
        self._after(st, su)
        self._dx("gate_proj", sched, self.z2, self.dgt, self.dz2a, st)
        self._dx("up_proj", sched, self.z2, self.du, self.dz2b, su)
        self._after(su, st)
        C.catq_rmsnorm_bwd(self.h, self.gamma2, self.r2, self.dz2a, self.dh, dZ2=self.dz2b, d_residual=self.d_out,
                           stream=st)
        self._dw("o_proj", sched, self.a, self.dh, grads)
        self._dx("o_proj", sched, self.a, self.dh, self.da, st)
        C.catq_attention_bwd(self.q, self.k, self.v, self.a, self.da, self.lse, self.delta, self.dq, self.dk, self.dv,
                             sh.B, sh.S, sh.n_heads, sh.n_kv_heads, sh.d, stream=st)
        self._dw("v_proj", sched, self.z1, self.dv, grads)
        for name, dy, pre, norm, r, nh in (("k_proj", self.dk, "kp", self.k_norm, "rk", sh.n_kv_heads),
                                           ("q_proj", self.dq, "qp", self.q_norm, "rq", sh.n_heads)):
            C.catq_rope(dy, sh.S, nh, sh.d, sh.base, inverse=True, stream=st)
            if norm is not None:  # through the head norm, in place
                C.catq_rmsnorm_bwd(getattr(self, pre).view(-1, sh.d), norm, getattr(self, r), dy.view(-1, sh.d),
                                   dy.view(-1, sh.d), stream=st)
            self._dw(name, sched, self.z1, dy, grads)
        self._join()
        return out

    def _dx(self, name, sched, X, dY, dX, stream):
        C.catq_soft_ternary_linear_bwd(self.layers[name], sched, X, dY, dX, stream=stream)

    def _dw(self, name, sched, X, dY, grads):
        """Linear `name`'s factor gradients on the next dW stream (in turn), after the work
        issued so far on the main stream, with that stream's workspace."""
        g = grads[name]
        sd, ws = self._dw_lane(self._next_side)
        self._next_side += 1
        self._after(self._main(), sd)
        C.catq_soft_ternary_linear_bwd(self.layers[name], sched, X, dY, None, g[0], g[1], g[2], workspace=ws,
                                       stream=sd)
