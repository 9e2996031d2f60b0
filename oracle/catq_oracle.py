"""Plain fp64 CPU oracle of the CAT-Q soft-ternary calibration hot path.

TEST INFRASTRUCTURE ONLY.  This module is imported by ``tests/``, by
``__graft_entry__.smoke()`` and by ``bench.py``'s CPU-baseline leg, and by nothing
else.  It shares no code with the CUDA path and never reads anything the CUDA path
produced.  Every function is the paper's definition written out in fp64 numpy, in the
paper's order and notation; matrix products use numpy's matmul as a library step.

Notation (CAT-Q, §2): W [N, K] is a linear layer's weight (row-major, out x in), X [M, K]
its calibration input, Y = X Wq^T its output.  W is flattened row-major and split into
G = N*K/g consecutive groups of g elements (App. B.2); every statistic and factor is per
group.

Pins (tests/test_oracle_pins.py) tie each function to something other than itself:
brute force, closed forms, limits and finite differences; the optimizer update also to
PyTorch's own AdamW; the 8-bit activation quantizer to exact grids, its error bound and a
brute-force nearest code.  One part is
"parity unpinned": the HARD-phase factor gradients (see ``linear_bwd``), which rest on
this library's reading of §2.3's stage-2 rule and have no independent reference.
"""
from __future__ import annotations

import numpy as np

PHASE_TEACHER, PHASE_SOFT, PHASE_HARD = 0, 1, 2
THR_HALF, THR_TWN07, THR_ABSMEAN, THR_TWN_STATIC = 0, 1, 2, 3


def _groups(W: np.ndarray, g: int) -> np.ndarray:
    """Row-major flatten and split into [G, g] (App. B.2: flattened, non-overlapping
    groups of size g)."""
    W = np.asarray(W, dtype=np.float64)
    assert W.size % g == 0
    return W.reshape(-1, g)


def group_stats(W: np.ndarray, g: int, thr_init: int = THR_HALF):
    """Eq. 3's frozen statistics per group and the initial threshold of §2.2.

    mu0 = mean of the group; alpha0 = mean |W - mu0|.  Delta0 = 0.5 in What units
    (§2.2 default) or, for the TWN rule of §2.2, the threshold 0.7 * mean|W| expressed
    in What units at identity factors: 0.7 * mean|W| / alpha0.

    The static approximations §2.2 starts from, as base statistics for the modulation
    (mu0 = 0, What = W / alpha):
      THR_ABSMEAN     (BitNet b1.58 and others): alpha0 = mean |W|, Delta = alpha / 2, so
                      Delta0 = 0.5 (alpha0 = 0: Delta0 = 0.5);
      THR_TWN_STATIC  (TWN): Delta_W = 0.7 mean |W|, alpha0 = mean of |W_i| over
                      |W_i| > Delta_W, Delta0 = Delta_W / alpha0 (alpha0 = 0, no element
                      above the threshold: Delta0 = 0.5).
    """
    Wg = _groups(W, g)
    if thr_init in (THR_ABSMEAN, THR_TWN_STATIC):
        mean_abs = np.abs(Wg).mean(axis=1)
        mu0 = np.zeros(Wg.shape[0])
        if thr_init == THR_ABSMEAN:
            return mu0, mean_abs, np.full_like(mean_abs, 0.5)
        dW = 0.7 * mean_abs
        above = np.abs(Wg) > dW[:, None]
        cnt = above.sum(axis=1)
        alpha0 = np.where(cnt > 0, (np.abs(Wg) * above).sum(axis=1) / np.maximum(cnt, 1), 0.0)
        with np.errstate(divide="ignore", invalid="ignore"):
            delta0 = np.where(alpha0 > 0, dW / np.where(alpha0 > 0, alpha0, 1.0), 0.5)
        return mu0, alpha0, delta0
    mu0 = Wg.mean(axis=1)
    alpha0 = np.abs(Wg - mu0[:, None]).mean(axis=1)
    if thr_init == THR_HALF:
        delta0 = np.full_like(mu0, 0.5)
    elif thr_init == THR_TWN07:
        mean_abs = np.abs(Wg).mean(axis=1)
        with np.errstate(divide="ignore", invalid="ignore"):
            delta0 = np.where(alpha0 > 0, 0.7 * mean_abs / np.where(alpha0 > 0, alpha0, 1.0), 0.5)
    else:
        raise ValueError("thr_init")
    return mu0, alpha0, delta0


def modulation(mu0, alpha0, delta0, d_mu, d_alpha, d_delta):
    """Eq. 3 and the threshold rule of §2.2:
    mu = mu0 + d_mu * alpha0, alpha = d_alpha * alpha0, Delta = d_delta * Delta0."""
    mu0, alpha0, delta0 = (np.asarray(a, np.float64) for a in (mu0, alpha0, delta0))
    d_mu, d_alpha, d_delta = (np.asarray(a, np.float64) for a in (d_mu, d_alpha, d_delta))
    mu = mu0 + d_mu * alpha0
    alpha = d_alpha * alpha0
    Delta = d_delta * delta0
    return mu, alpha, Delta


def transformed_weight(W, g, mu, alpha):
    """Eq. 3: What = (W - mu) / alpha, per group, returned as [G, g].
    A group with alpha == 0 is degenerate; its What is set to 0 (library reading)."""
    Wg = _groups(W, g)
    safe = np.where(alpha != 0, alpha, 1.0)
    What = (Wg - mu[:, None]) / safe[:, None]
    return np.where((alpha != 0)[:, None], What, 0.0)


def transition_f(x, s, Delta):
    """Eq. 5: f(x; s, Delta) = [tanh(s(x - Delta)) + tanh(s(x + Delta))] / (2 tanh s)."""
    x = np.asarray(x, np.float64)
    return (np.tanh(s * (x - Delta)) + np.tanh(s * (x + Delta))) / (2.0 * np.tanh(s))


def transition_f_grads(x, s, Delta):
    """Partial derivatives of Eq. 5 with respect to its input x and to Delta:
    with a = tanh(s(x-Delta)), b = tanh(s(x+Delta)) and c = 2 tanh s,
    df/dx = s [(1 - a^2) + (1 - b^2)] / c,  df/dDelta = s [(1 - b^2) - (1 - a^2)] / c."""
    x = np.asarray(x, np.float64)
    a = np.tanh(s * (x - Delta))
    b = np.tanh(s * (x + Delta))
    c = 2.0 * np.tanh(s)
    dfdx = s * ((1.0 - a * a) + (1.0 - b * b)) / c
    dfdD = s * ((1.0 - b * b) - (1.0 - a * a)) / c
    return dfdx, dfdD


def hard_q(x, Delta):
    """Eq. 2: Q(x; Delta) = 1 if x > Delta, 0 if |x| <= Delta, -1 if x < -Delta."""
    x = np.asarray(x, np.float64)
    return np.where(x > Delta, 1.0, np.where(x < -Delta, -1.0, 0.0))


def _per_elem(v, g):
    return np.repeat(np.asarray(v, np.float64), g)


def ternary_weight(W, g, stats, factors, phase, s, with_mu=False):
    """Eq. 6 and the reconstruction W ~ alpha T without mu (§2.2, App. B.2), or with it,
    W ~ alpha T + mu, when `with_mu` (the variant of the tab:mu ablation).

    Returns (Wq [N, K], T [N, K], What [N, K], alpha [G], Delta [G]).
    TEACHER (t = 0): T = W and Wq = W.  SOFT: T = f(What; s, Delta).  HARD: T = Q(What; Delta).
    """
    W = np.asarray(W, np.float64)
    N, K = W.shape
    mu, alpha, Delta = modulation(*stats, *factors)
    What = transformed_weight(W, g, mu, alpha)
    if phase == PHASE_TEACHER:
        return W.copy(), W.copy(), What.reshape(N, K), alpha, Delta
    if phase == PHASE_SOFT:
        T = transition_f(What, s, Delta[:, None])
    elif phase == PHASE_HARD:
        T = hard_q(What, Delta[:, None])
    else:
        raise ValueError("phase")
    T = np.where((alpha != 0)[:, None], T, 0.0)
    Wq = alpha[:, None] * T
    if with_mu:
        Wq = Wq + mu[:, None]  # a group with alpha == 0 reconstructs as mu
    return Wq.reshape(N, K), T.reshape(N, K), What.reshape(N, K), alpha, Delta


def linear_fwd(X, Wq):
    """The contraction of one linear: Y = X Wq^T (Y [M, N], X [M, K], Wq [N, K])."""
    return np.asarray(X, np.float64) @ np.asarray(Wq, np.float64).T


def recon_loss(Y, Y_ref, reduction: int = 0):
    """Eq. 7 for one linear: the squared L2 distance between the quantized output and the
    full-precision (teacher) output, averaged over elements (reduction 0, the library
    default) or summed (1).  Returns (loss, dL/dY)."""
    d = np.asarray(Y, np.float64) - np.asarray(Y_ref, np.float64)
    if reduction == 0:
        n = d.size
        return float((d * d).sum() / n), 2.0 * d / n
    return float((d * d).sum()), 2.0 * d


def factor_grads_from_G(Gw, W, g, stats, factors, phase, s, with_mu=False):
    """Chain rule of Eq. 3 and Eq. 5/6 from G = dL/dWq [N, K] into the three factors.

    Wq = alpha * T(What), What = (W - mu)/alpha, mu = mu0 + d_mu*alpha0,
    alpha = d_alpha*alpha0, Delta = d_delta*Delta0 give per element
      dWq/dmu = -f'(What),  dWq/dalpha = T - What f'(What),  dWq/dDelta = alpha df/dDelta,
    and the factor gradients are the group sums times alpha0, alpha0 and Delta0.
    SOFT: T = f.  HARD (reading of §2.3's stage-2 rule): T = Q(What; Delta) as in the
    forward, with f's derivatives at the given s — parity unpinned.  TEACHER: zeros.
    With mu in the reconstruction (Wq = alpha T + mu), dWq/dmu = 1 - f'(What).
    """
    mu0, alpha0, delta0 = (np.asarray(a, np.float64) for a in stats)
    G = mu0.shape[0]
    if phase == PHASE_TEACHER:
        z = np.zeros(G)
        return z, z.copy(), z.copy()
    mu, alpha, Delta = modulation(*stats, *factors)
    What = transformed_weight(W, g, mu, alpha)
    Gg = np.asarray(Gw, np.float64).reshape(-1, g)
    dfdx, dfdD = transition_f_grads(What, s, Delta[:, None])
    if phase == PHASE_SOFT:
        T = transition_f(What, s, Delta[:, None])
    elif phase == PHASE_HARD:
        T = hard_q(What, Delta[:, None])
    else:
        raise ValueError("phase")
    live = alpha != 0
    c_mu = (1.0 - dfdx) if with_mu else -dfdx
    g_dmu = np.where(live, alpha0 * (Gg * c_mu).sum(axis=1), 0.0)
    g_dalpha = np.where(live, alpha0 * (Gg * (T - What * dfdx)).sum(axis=1), 0.0)
    g_ddelta = np.where(live, delta0 * alpha * (Gg * dfdD).sum(axis=1), 0.0)
    return g_dmu, g_dalpha, g_ddelta


def linear_bwd(X, dY, W, g, stats, factors, phase, s, with_mu=False):
    """Backward of Y = X Wq^T: dX = dY Wq, G = dY^T X (= dL/dWq), then the factor
    gradients of ``factor_grads_from_G``.  Returns (dX, g_dmu, g_dalpha, g_ddelta)."""
    X = np.asarray(X, np.float64)
    dY = np.asarray(dY, np.float64)
    Wq = ternary_weight(W, g, stats, factors, phase, s, with_mu)[0]
    dX = dY @ Wq
    Gw = dY.T @ X
    return (dX,) + factor_grads_from_G(Gw, W, g, stats, factors, phase, s, with_mu)


def calibration_step(X, W, g, stats, factors, phase, s, reduction=0, with_mu=False):
    """One soft-ternary calibration step for one linear (Eq. 6, Eq. 7): teacher output,
    quantized output, loss, and every gradient.  Returns a dict."""
    Y_ref = linear_fwd(X, W)
    Wq = ternary_weight(W, g, stats, factors, phase, s, with_mu)[0]
    Y = linear_fwd(X, Wq)
    loss, dY = recon_loss(Y, Y_ref, reduction)
    dX, g_dmu, g_dalpha, g_ddelta = linear_bwd(X, dY, W, g, stats, factors, phase, s, with_mu)
    return dict(Y_ref=Y_ref, Y=Y, loss=loss, dY=dY, dX=dX, g_dmu=g_dmu, g_dalpha=g_dalpha,
                g_ddelta=g_ddelta, Wq=Wq)


def act_quant_a8(X):
    """Per-token symmetric 8-bit quantization of a linear's input, the activation side of
    the W1.58A8 setting (§1, App. B.2; the paper does not state the quantizer, and this is
    the reading of dynamic per-token absmax quantization):
        scale_m = max_k |X[m, k]| / 127,   q[m, k] = clamp(round(X[m, k] / scale_m), -127, 127)
    with round-half-to-even, and scale 0 with q = 0 for a row of zeros.  Because the scale
    and the quotient decide integer codes, both are taken in fp32 with IEEE division (the
    precision of the kernel); everything after them is fp64.
    Returns (q [M, K] int64, scale [M] float32)."""
    X32 = np.asarray(X, np.float32)
    amax = np.abs(X32).max(axis=1)
    scale = (amax / np.float32(127.0)).astype(np.float32)
    safe = np.where(scale > 0, scale, np.float32(1.0)).astype(np.float32)
    q = np.clip(np.rint(X32 / safe[:, None]), -127, 127)
    q[scale == 0] = 0
    return q.astype(np.int64), scale


def a8_calibration_step(X, W, g, stats, factors, phase, s, reduction=0, with_mu=False):
    """One calibration step of a linear whose input is quantized to 8 bits per token
    (``act_quant_a8``): the teacher is the full-precision output X W^T (Eq. 7's F(W, X)),
    the quantized output Y = X_q Wq^T with X_q = scale q; the rounding passes gradients
    straight through, so dX = dY Wq, and G = dY^T X_q is the gradient of Wq.  Returns the
    dict of ``calibration_step`` plus q, scale and X_q."""
    q, scale = act_quant_a8(X)
    Xq = q.astype(np.float64) * scale.astype(np.float64)[:, None]
    Y_ref = linear_fwd(X, W)
    Wq = ternary_weight(W, g, stats, factors, phase, s, with_mu)[0]
    Y = linear_fwd(Xq, Wq)
    loss, dY = recon_loss(Y, Y_ref, reduction)
    dX, g_dmu, g_dalpha, g_ddelta = linear_bwd(Xq, dY, W, g, stats, factors, phase, s, with_mu)
    return dict(Y_ref=Y_ref, Y=Y, loss=loss, dY=dY, dX=dX, g_dmu=g_dmu, g_dalpha=g_dalpha,
                g_ddelta=g_ddelta, Wq=Wq, q=q, scale=scale, Xq=Xq)


def hard_codes(W, g, stats, factors):
    """Eq. 4: T = Q(What; d_delta * Delta0) as int8, plus alpha per group and the fp64
    distance of every |What| from its threshold (for the near-threshold listing)."""
    mu, alpha, Delta = modulation(*stats, *factors)
    What = transformed_weight(W, g, mu, alpha)
    T = hard_q(What, Delta[:, None])
    T = np.where((alpha != 0)[:, None], T, 0.0).astype(np.int8)
    gap = np.abs(np.abs(What) - Delta[:, None])
    rel_gap = gap / np.where(Delta != 0, np.abs(Delta), 1.0)[:, None]
    return T.reshape(-1), alpha, rel_gap.reshape(-1)


def pack_codes(T):
    """2-bit packing of ternary codes (this library's encoding; the paper fixes none):
    element e stores T_e + 1 in bits [2*(e % 4), 2*(e % 4) + 1] of byte e // 4."""
    T = np.asarray(T).reshape(-1).astype(np.int64)
    assert T.size % 4 == 0
    out = np.zeros(T.size // 4, dtype=np.int64)
    for i in range(4):
        out |= (T[i::4] + 1) << (2 * i)
    return out.astype(np.uint8)


def ternary_infer(codes, alpha, N, K, g, X, mu=None):
    """Inference with the deployed form of a calibrated layer: App. B.2 keeps only the
    ternary codes T and the group scale alpha (W ~ alpha T, Eq. 4), so Y = X (alpha T)^T
    with T read from the 2-bit codes (``pack_codes``'s layout) and alpha [G] per group of g
    consecutive elements of a row.  With the group offsets mu [G] of the W ~ alpha T + mu
    variant, Y = X (alpha T + mu)^T.  Returns Y [M, N] in fp64."""
    T = unpack_codes(codes, N * K).astype(np.float64).reshape(N, K)
    Wq = T * _per_elem(alpha, g).reshape(N, K)
    if mu is not None:
        Wq = Wq + _per_elem(mu, g).reshape(N, K)
    return linear_fwd(X, Wq)


def unpack_codes(codes, n):
    """Inverse of ``pack_codes`` (used only by tests)."""
    codes = np.asarray(codes, np.uint8).astype(np.int64)
    T = np.zeros(codes.size * 4, dtype=np.int64)
    for i in range(4):
        T[i::4] = ((codes >> (2 * i)) & 3) - 1
    return T[:n].astype(np.int8)


# ------------------------------------------------------------------ calibration schedule and update
# App. B.1 fixes the optimizer (AdamW), the epochs (m = 60), the learning rate of the
# modulation factors (1e-3) with a linear decay to zero, gamma = 0.8 and s0 = 30; §2.3 maps
# the normalised epoch t to Eq. 6's branch and sharpness.

def schedule_at_epoch(e: int, m: int, gamma: float, s0: float):
    """Eq. 6's schedule point of calibration epoch e of m: t = e / m; t = 0 is the teacher
    branch, 0 < t <= gamma the soft stage with s = (t / gamma) s0, gamma < t <= 1 the hard
    stage.  The comparison t <= gamma is made as e <= floor(gamma m + 1e-9), so that
    gamma m = 48 at the paper's defaults counts 48 soft epochs whatever the rounding of
    0.8 * 60.  The hard stage's backward keeps the sharpness of the last soft epoch (§2.3:
    the gradients of the last iteration of the first stage), i.e. (t_last / gamma) s0 with
    t_last = floor(gamma m) / m; that is s0 when gamma m is an integer (the paper's
    defaults) and below s0 otherwise.  With no soft epoch at all (gamma m < 1) there is no
    last soft sharpness, and s0 is used.
    Returns (phase, s)."""
    assert 0 <= e <= m and m >= 1 and 0.0 < gamma <= 1.0 and s0 > 0.0
    if e == 0:
        return PHASE_TEACHER, 0.0
    soft_epochs = int(np.floor(gamma * m + 1e-9))
    if e <= soft_epochs:
        t = e / m
        return PHASE_SOFT, (t / gamma) * s0
    if soft_epochs == 0:
        return PHASE_HARD, float(s0)
    t_last = soft_epochs / m
    return PHASE_HARD, (t_last / gamma) * s0


def linear_decay_lr(lr0: float, k: int, total: int) -> float:
    """Learning rate of update k (0-based) of `total` under App. B.1's linear decay to zero:
    lr0 (1 - k / total), which reaches zero one update after the last."""
    assert 0 <= k < total
    return lr0 * (1.0 - k / total)


def adamw_step(p, grad, m, v, t: int, lr: float, beta1: float = 0.9, beta2: float = 0.999,
               eps: float = 1e-8, weight_decay: float = 0.0):
    """One AdamW update of parameters p (Loshchilov & Hutter, "Decoupled weight decay
    regularization": the decay acts on p directly, not through the gradient) with Adam's
    bias-corrected moments (Kingma & Ba), update count t >= 1.  The decay is scaled by the
    learning rate, the PyTorch convention.  In order:
        p <- p - lr * weight_decay * p
        m <- beta1 m + (1 - beta1) grad,   v <- beta2 v + (1 - beta2) grad^2
        p <- p - lr * m_hat / (sqrt(v_hat) + eps),  m_hat = m / (1 - beta1^t),
                                                      v_hat = v / (1 - beta2^t)
    Returns (p, m, v) as new fp64 arrays."""
    p = np.asarray(p, np.float64)
    grad = np.asarray(grad, np.float64)
    m = np.asarray(m, np.float64)
    v = np.asarray(v, np.float64)
    p = p - lr * weight_decay * p
    m = beta1 * m + (1.0 - beta1) * grad
    v = beta2 * v + (1.0 - beta2) * grad * grad
    m_hat = m / (1.0 - beta1 ** t)
    v_hat = v / (1.0 - beta2 ** t)
    p = p - lr * m_hat / (np.sqrt(v_hat) + eps)
    return p, m, v


def project_factors(d_mu, d_alpha, d_delta, margin: float):
    """§2.2's constraints -1 < d_mu < 1, d_alpha > 0, d_delta > 0, enforced as the Euclidean
    projection onto the closed sets [-1 + margin, 1 - margin], [margin, inf), [margin, inf)
    (the paper does not say how they are kept; NaN stays NaN)."""
    return (np.clip(np.asarray(d_mu, np.float64), -1.0 + margin, 1.0 - margin),
            np.clip(np.asarray(d_alpha, np.float64), margin, np.inf),
            np.clip(np.asarray(d_delta, np.float64), margin, np.inf))


def factor_update(factors, grads, moments, t: int, lr: float, beta1: float = 0.9, beta2: float = 0.999,
                  eps: float = 1e-8, weight_decay: float = 0.0, margin: float = 1e-4):
    """The update after a calibration step: AdamW on each of (d_mu, d_alpha, d_delta) with
    its gradient, then the projection of ``project_factors``.  moments = (m_mu, m_alpha,
    m_delta, v_mu, v_alpha, v_delta).  Returns (factors, moments) as tuples of fp64 arrays."""
    new_p, new_m, new_v = [], [], []
    for q in range(3):
        p, m, v = adamw_step(factors[q], grads[q], moments[q], moments[3 + q], t, lr, beta1, beta2, eps,
                             weight_decay)
        new_p.append(p)
        new_m.append(m)
        new_v.append(v)
    return project_factors(*new_p, margin), tuple(new_m) + tuple(new_v)


# ------------------------------------------------------------------ direct learning and Fig. fig:error
# §2.2 compares three ways to set a group's alpha and Delta: a static approximation (SA, the
# absmean rule of BitNet b1.58 and others), learning alpha and Delta directly (DL, started
# from that static rule), and the learnable modulation (LM); Fig. fig:error plots the
# per-group weight reconstruction error each leaves.

def direct_grads(d_alpha, d_delta, g_dalpha, g_ddelta):
    """Gradients of direct learning's parameters from the modulation's factor gradients.
    DL learns the scale alpha and the weight-space threshold Delta_W = alpha Delta of each
    group, with mu fixed at mu0 (0 for the static rules), read here in units of the group's
    static statistics so that the paper's learning rate means the same relative step as for
    the modulation's factors:
        a = alpha / alpha0 = d_alpha,   d = Delta_W / (alpha0 Delta0) = d_alpha d_delta.
    With d_alpha = a and d_delta = d / a the chain rule gives
        dL/da = g_dalpha - g_ddelta d_delta / d_alpha,   dL/dd = g_ddelta / d_alpha."""
    d_alpha = np.asarray(d_alpha, np.float64)
    d_delta = np.asarray(d_delta, np.float64)
    g_dalpha = np.asarray(g_dalpha, np.float64)
    g_ddelta = np.asarray(g_ddelta, np.float64)
    return g_dalpha - g_ddelta * d_delta / d_alpha, g_ddelta / d_alpha


def direct_update(d_alpha, d_delta, g_dalpha, g_ddelta, moments, t: int, lr: float, beta1: float = 0.9,
                  beta2: float = 0.999, eps: float = 1e-8, weight_decay: float = 0.0, margin: float = 1e-4):
    """One update of direct learning: AdamW (``adamw_step``) on a = d_alpha and
    d = d_alpha d_delta with the gradients of ``direct_grads``, the constraints alpha > 0 and
    Delta > 0 kept as a >= margin and d >= margin, then d_alpha = a and d_delta = d / a.
    moments = (m_a, m_d, v_a, v_d).  Returns (d_alpha, d_delta, moments)."""
    d_alpha = np.asarray(d_alpha, np.float64)
    d_delta = np.asarray(d_delta, np.float64)
    ga, gd = direct_grads(d_alpha, d_delta, g_dalpha, g_ddelta)
    a, ma, va = adamw_step(d_alpha, ga, moments[0], moments[2], t, lr, beta1, beta2, eps, weight_decay)
    d, md, vd = adamw_step(d_alpha * d_delta, gd, moments[1], moments[3], t, lr, beta1, beta2, eps, weight_decay)
    a = np.clip(a, margin, np.inf)
    d = np.clip(d, margin, np.inf)
    return a, d / a, (ma, md, va, vd)


def group_recon_error(W, g, stats, factors):
    """Per-group weight reconstruction error of the hard ternarization (Fig. fig:error):
    the mean over the group of (W - alpha Q(What; Delta))^2 (W ~ alpha T, no mu)."""
    Wq = ternary_weight(W, g, stats, factors, PHASE_HARD, 1.0)[0]
    d = (np.asarray(W, np.float64) - Wq).reshape(-1, g)
    return (d * d).mean(axis=1)


# ------------------------------------------------------------------ one decoder block (§2.4)
# Eq. 7 reconstructs the output of a window of layers.  The window here is one decoder block
# of the Llama / Qwen family (pre-norm, grouped-query causal attention with rotary position
# embedding, SwiGLU MLP), all seven linears soft-ternary, the teacher the same block with
# full-precision weights.  Tokens are rows t = b S + s of a [B S, H] activation.

def rmsnorm(x, gamma, eps):
    """RMSNorm of each row: y = gamma * x / sqrt(mean(x^2) + eps).  Returns (y, r) with
    r = 1 / sqrt(mean(x^2) + eps) per row."""
    x = np.asarray(x, np.float64)
    r = 1.0 / np.sqrt((x * x).mean(axis=1) + eps)
    return x * r[:, None] * np.asarray(gamma, np.float64)[None, :], r


def rmsnorm_bwd(x, gamma, r, dy):
    """Gradient of ``rmsnorm`` with respect to x: with u = gamma * dy,
    dx = r u - x r^3 mean(u x)."""
    x = np.asarray(x, np.float64)
    u = np.asarray(dy, np.float64) * np.asarray(gamma, np.float64)[None, :]
    return r[:, None] * u - x * (r ** 3 * (u * x).mean(axis=1))[:, None]


def rope(x, S, n_heads, d, base, inverse=False):
    """Rotary position embedding of each head of x [B S, n_heads d] (the half-split pairing:
    element i and i + d/2 of a head rotate together) by the angle s base^(-2i/d) of the
    token's position s; ``inverse`` rotates back (the gradient of the rotation)."""
    x = np.asarray(x, np.float64)
    T = x.shape[0]
    pos = (np.arange(T) % S).astype(np.float64)
    inv_freq = base ** (-2.0 * np.arange(d // 2) / d)
    ang = pos[:, None] * inv_freq[None, :]
    c, s_ = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    if inverse:
        s_ = -s_
    xh = x.reshape(T, n_heads, d)
    a, b = xh[..., : d // 2], xh[..., d // 2:]
    return np.concatenate([a * c - b * s_, a * s_ + b * c], axis=2).reshape(T, n_heads * d)


def attention(q, k, v, B, S, nh, nkv, d):
    """Causal grouped-query attention: head h uses key/value head h // (nh / nkv);
    O = softmax(Q K^T / sqrt(d), keys <= query) V per batch and head.  Returns (o [B S, nh d],
    P [B, nh, S, S] the attention probabilities)."""
    q = np.asarray(q, np.float64).reshape(B, S, nh, d)
    k = np.asarray(k, np.float64).reshape(B, S, nkv, d)
    v = np.asarray(v, np.float64).reshape(B, S, nkv, d)
    rep = nh // nkv
    kh = np.repeat(k, rep, axis=2)
    vh = np.repeat(v, rep, axis=2)
    s = np.einsum("bqhd,bkhd->bhqk", q, kh) / np.sqrt(d)
    s = np.where(np.tril(np.ones((S, S), bool))[None, None], s, -np.inf)
    s = s - s.max(axis=3, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=3, keepdims=True)
    o = np.einsum("bhqk,bkhd->bqhd", p, vh)
    return o.reshape(B * S, nh * d), p


def attention_bwd(q, k, v, p, do, B, S, nh, nkv, d):
    """Gradients of ``attention``: with dS = P (dP - rowsum(dP P)), dP = dO V^T,
    dQ = dS K / sqrt(d), dK = dS^T Q / sqrt(d), dV = P^T dO, the key/value gradients summed
    over the heads that share them."""
    q = np.asarray(q, np.float64).reshape(B, S, nh, d)
    k = np.asarray(k, np.float64).reshape(B, S, nkv, d)
    v = np.asarray(v, np.float64).reshape(B, S, nkv, d)
    do = np.asarray(do, np.float64).reshape(B, S, nh, d)
    rep = nh // nkv
    kh = np.repeat(k, rep, axis=2)
    vh = np.repeat(v, rep, axis=2)
    dp = np.einsum("bqhd,bkhd->bhqk", do, vh)
    ds = p * (dp - (dp * p).sum(axis=3, keepdims=True))
    dq = np.einsum("bhqk,bkhd->bqhd", ds, kh) / np.sqrt(d)
    dkh = np.einsum("bhqk,bqhd->bkhd", ds, q) / np.sqrt(d)
    dvh = np.einsum("bhqk,bqhd->bkhd", p, do)
    dk = dkh.reshape(B, S, nkv, rep, d).sum(axis=3)
    dv = dvh.reshape(B, S, nkv, rep, d).sum(axis=3)
    return dq.reshape(B * S, nh * d), dk.reshape(B * S, nkv * d), dv.reshape(B * S, nkv * d)


def attention_logsumexp(q, k, B, S, nh, nkv, d):
    """The softmax normaliser of ``attention``: for every sequence, head and query s, the
    natural log of the sum over keys s' <= s of exp(q . k / sqrt(d)); [B, nh, S]."""
    q = np.asarray(q, np.float64).reshape(B, S, nh, d)
    k = np.repeat(np.asarray(k, np.float64).reshape(B, S, nkv, d), nh // nkv, axis=2)
    s = np.einsum("bqhd,bkhd->bhqk", q, k) / np.sqrt(d)
    s = np.where(np.tril(np.ones((S, S), bool))[None, None], s, -np.inf)
    m = s.max(axis=3)
    return m + np.log(np.exp(s - m[..., None]).sum(axis=3))


def silu(a):
    a = np.asarray(a, np.float64)
    return a / (1.0 + np.exp(-a))


def swiglu(gt, u):
    """The SwiGLU MLP's gate: silu(gt) * u elementwise."""
    return silu(gt) * np.asarray(u, np.float64)


def swiglu_bwd(gt, u, dm):
    """Gradients of ``swiglu`` from dm: with sigma the logistic function,
    d_gt = dm u sigma(gt) (1 + gt (1 - sigma(gt))) and d_u = dm silu(gt)."""
    gt, u, dm = (np.asarray(a, np.float64) for a in (gt, u, dm))
    sg = 1.0 / (1.0 + np.exp(-gt))
    return dm * u * sg * (1.0 + gt * (1.0 - sg)), dm * silu(gt)


BLOCK_LINEARS = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def _head_norm(x, gamma, d, eps):
    """RMSNorm of every head (rows of d elements) of x [T, heads d]; returns (y, r per head)."""
    y, r = rmsnorm(np.asarray(x, np.float64).reshape(-1, d), gamma, eps)
    return y.reshape(np.shape(x)), r


def block_forward(x, Wq, gamma1, gamma2, B, S, nh, nkv, d, base, eps, q_norm=None, k_norm=None):
    """One decoder block with the effective weights Wq[name] ([N, K] each):
    z1 = RMSNorm(x); q, k, v = z1 W^T; (Qwen3: RMSNorm of every query and key head with the
    weights q_norm, k_norm [d]); rotary q, k; a = attention; h = x + a Wo^T;
    z2 = RMSNorm(h); m = silu(z2 Wg^T) * (z2 Wu^T); out = h + m Wd^T.  Returns (out, cache)."""
    x = np.asarray(x, np.float64)
    z1, r1 = rmsnorm(x, gamma1, eps)
    qp, kp = linear_fwd(z1, Wq["q_proj"]), linear_fwd(z1, Wq["k_proj"])
    qn, rq = _head_norm(qp, q_norm, d, eps) if q_norm is not None else (qp, None)
    kn, rk = _head_norm(kp, k_norm, d, eps) if k_norm is not None else (kp, None)
    q = rope(qn, S, nh, d, base)
    k = rope(kn, S, nkv, d, base)
    v = linear_fwd(z1, Wq["v_proj"])
    a, p = attention(q, k, v, B, S, nh, nkv, d)
    h = x + linear_fwd(a, Wq["o_proj"])
    z2, r2 = rmsnorm(h, gamma2, eps)
    gt = linear_fwd(z2, Wq["gate_proj"])
    u = linear_fwd(z2, Wq["up_proj"])
    m = swiglu(gt, u)
    out = h + linear_fwd(m, Wq["down_proj"])
    return out, dict(z1=z1, qp=qp, kp=kp, rq=rq, rk=rk, q=q, k=k, v=v, a=a, p=p, h=h, z2=z2, r2=r2, gt=gt, u=u,
                     m=m)


def block_calibration_step(x, W, g, stats, factors, gamma1, gamma2, B, S, nh, nkv, d, base, eps, phase, s,
                           reduction=0, q_norm=None, k_norm=None):
    """One calibration step of a window of one decoder block (Eq. 7 over the block output):
    the teacher block with full-precision weights, the block with each linear's Eq. 6 weight
    (W, stats, factors: dicts by linear name), the loss, and every linear's factor gradients
    through the block's backward.  The block input is fixed (the window's input), so no
    gradient flows into x.  Returns a dict: out, out_ref, loss, and g[name] = (g_dmu,
    g_dalpha, g_ddelta)."""
    Wq = {n: ternary_weight(W[n], g, stats[n], factors[n], phase, s)[0] for n in BLOCK_LINEARS}
    out_ref, _ = block_forward(x, {n: np.asarray(W[n], np.float64) for n in BLOCK_LINEARS}, gamma1, gamma2, B,
                               S, nh, nkv, d, base, eps, q_norm, k_norm)
    out, c = block_forward(x, Wq, gamma1, gamma2, B, S, nh, nkv, d, base, eps, q_norm, k_norm)
    loss, d_out = recon_loss(out, out_ref, reduction)
    G = {}

    def grads(name, X, dY):
        G[name] = factor_grads_from_G(np.asarray(dY).T @ np.asarray(X), W[name], g, stats[name], factors[name],
                                      phase, s)

    grads("down_proj", c["m"], d_out)
    dm = d_out @ Wq["down_proj"]
    d_gt, d_u = swiglu_bwd(c["gt"], c["u"], dm)
    grads("gate_proj", c["z2"], d_gt)
    grads("up_proj", c["z2"], d_u)
    dz2 = d_gt @ Wq["gate_proj"] + d_u @ Wq["up_proj"]
    dh = d_out + rmsnorm_bwd(c["h"], gamma2, c["r2"], dz2)
    grads("o_proj", c["a"], dh)
    da = dh @ Wq["o_proj"]
    dq, dk, dv = attention_bwd(c["q"], c["k"], c["v"], c["p"], da, B, S, nh, nkv, d)
    dq, dk = rope(dq, S, nh, d, base, inverse=True), rope(dk, S, nkv, d, base, inverse=True)
    if q_norm is not None:
        dq = rmsnorm_bwd(c["qp"].reshape(-1, d), q_norm, c["rq"], dq.reshape(-1, d)).reshape(dq.shape)
    if k_norm is not None:
        dk = rmsnorm_bwd(c["kp"].reshape(-1, d), k_norm, c["rk"], dk.reshape(-1, d)).reshape(dk.shape)
    grads("q_proj", c["z1"], dq)
    grads("k_proj", c["z1"], dk)
    grads("v_proj", c["z1"], dv)
    return dict(out=out, out_ref=out_ref, loss=loss, g=G, cache=c)
