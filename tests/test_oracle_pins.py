"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: exhaustive
enumeration, closed forms, limits stated in §2.3, special cases that reduce to a
textbook rule, and central finite differences.  A plausible slip in the oracle (a
dropped term, a flipped sign, a transposed operand, a wrong group index) fails at least
one of them.  No GPU is used.
"""
import itertools
import os

import numpy as np
import pytest

from oracle import catq_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- Eq. 1 / Eq. 2 (brute force)

def _half_enum():
    """All 3^8 ternary vectors of length 8."""
    return np.array(list(itertools.product([-1, 0, 1], repeat=8)), dtype=np.float64)


@pytest.mark.parametrize("delta", [0.5, 0.3, 0.8])
def test_q_is_the_exhaustive_minimiser_4x4(delta):
    """For a fixed scale, Q(x; Delta) (Eq. 2) is the unique minimiser over all 3^16 ternary
    4x4 matrices of sum (x - T)^2 + (2 Delta - 1) ||T||_0: choosing +-1 over 0 costs
    (|x| - 1)^2 - x^2 + (2 Delta - 1) = 2 (Delta - |x|), negative iff |x| > Delta.  At
    Delta = 1/2 this is nearest-ternary rounding, i.e. argmin_T ||What - T||^2 with the
    paper's Delta0 = 0.5 in What units (§2.2)."""
    r = np.random.default_rng(7)
    half = _half_enum()
    for trial in range(3):
        x = r.uniform(-1.6, 1.6, 16)
        x[np.abs(np.abs(x) - delta) < 1e-3] += 0.01  # keep clear of exact ties
        pen = 2 * delta - 1
        a, b = x[:8], x[8:]
        cost_a = ((a[None, :] - half) ** 2).sum(1) + pen * (half != 0).sum(1)
        cost_b = ((b[None, :] - half) ** 2).sum(1) + pen * (half != 0).sum(1)
        best, arg = np.inf, None
        for i in range(half.shape[0]):  # exhaustive over all 3^16 pairs
            tot = cost_a[i] + cost_b
            j = int(np.argmin(tot))
            if tot[j] < best:
                best, arg = tot[j], (i, j)
        T_brute = np.concatenate([half[arg[0]], half[arg[1]]])
        np.testing.assert_array_equal(O.hard_q(x, delta), T_brute)


def test_twn_objective_brute_force_is_a_threshold_ternarization():
    """Eq. 1 solved by enumerating all 3^16 T for a 4x4 W (best alpha > 0 per T): the
    minimiser keeps the largest |W| with their signs, i.e. it is Q(W; Delta) (Eq. 2) for a
    threshold between the kept and the dropped magnitudes, and alpha is the mean |W| over
    the kept set (TWN's alpha, §2.2)."""
    r = np.random.default_rng(11)
    half = _half_enum()
    nnz_h = (half != 0).sum(1).astype(np.float64)
    for trial in range(3):
        W = r.standard_normal(16)
        a, b = W[:8], W[8:]
        dot_a, dot_b = half @ a, half @ b
        best, arg = np.inf, None
        for i in range(half.shape[0]):
            nnz = nnz_h[i] + nnz_h
            dot = dot_a[i] + dot_b
            with np.errstate(divide="ignore", invalid="ignore"):
                red = np.where((nnz > 0) & (dot > 0), dot * dot / np.where(nnz > 0, nnz, 1), 0.0)
            obj = (W * W).sum() - red  # min over alpha > 0 of ||W - alpha T||^2
            j = int(np.argmin(obj))
            if obj[j] < best:
                best, arg = obj[j], (i, j)
        T = np.concatenate([half[arg[0]], half[arg[1]]])
        kept = np.abs(W[T != 0])
        dropped = np.abs(W[T == 0])
        assert kept.size > 0
        lo = dropped.max() if dropped.size else 0.0
        delta = 0.5 * (lo + kept.min())
        np.testing.assert_array_equal(O.hard_q(W, delta), T)
        alpha = (W * T).sum() / (T != 0).sum()
        np.testing.assert_allclose(alpha, kept.mean(), rtol=1e-12)


def test_q_tie_goes_to_zero():
    """Eq. 2 uses |x| <= Delta for the zero state."""
    np.testing.assert_array_equal(O.hard_q(np.array([0.5, -0.5, 0.5000001, -0.5000001]), 0.5),
                                  [0, 0, 1, -1])


# ----------------------------------------------------------------- Eq. 5 (closed forms, limits)

@pytest.mark.parametrize("s", [1e-3, 0.625, 4.95, 30.0, 300.0])
def test_f_at_threshold_half_is_half(s):
    """f(1/2; s, 1/2) = [tanh 0 + tanh s] / (2 tanh s) = 1/2 for every s."""
    assert abs(O.transition_f(0.5, s, 0.5) - 0.5) < 1e-15


@pytest.mark.parametrize("s,D", [(0.625, 0.5), (15.0, 0.4), (30.0, 0.6)])
def test_f_is_odd(s, D):
    """Property (1) of §2.3: the curve is symmetric about the origin."""
    x = np.linspace(-3, 3, 601)
    np.testing.assert_allclose(O.transition_f(-x, s, D), -O.transition_f(x, s, D), atol=1e-15)


@pytest.mark.parametrize("D", [0.3, 0.5, 1.2])
def test_f_small_s_series(D):
    """Property (2) of §2.3 (s -> 0 gives the identity), to second order: expanding tanh
    gives f(x) = x - s^2 x (x^2 + 3 Delta^2 - 1) / 3 + O(s^4)."""
    s = 1e-4
    x = np.linspace(-2, 2, 41)
    corr = -(s * s) * x * (x * x + 3 * D * D - 1) / 3  # ~1e-8; the O(s^4) rest is ~1e-16
    np.testing.assert_allclose(O.transition_f(x, s, D) - x, corr, atol=2e-13)
    np.testing.assert_allclose(O.transition_f(x, 1e-6, D), x, atol=1e-11)


@pytest.mark.parametrize("D", [0.3, 0.5, 0.9])
def test_f_hard_limit_is_q(D):
    """Property (4) of §2.3: s -> infinity gives Q (Eq. 2) away from |x| = Delta; scaled by
    alpha the outputs lie in {-alpha, 0, alpha}; at |x| = Delta the limit is +-1/2."""
    s = 1e5
    x = np.linspace(-3, 3, 6001)
    x = x[np.abs(np.abs(x) - D) > 1e-3]
    f = O.transition_f(x, s, D)
    np.testing.assert_allclose(f, O.hard_q(x, D), atol=1e-12)
    alpha = 0.037
    vals = np.unique(np.round(alpha * f / alpha * 1e9) / 1e9)
    assert set(vals.tolist()) <= {-1.0, 0.0, 1.0}
    np.testing.assert_allclose(O.transition_f(np.array([D, -D]), s, D), [0.5, -0.5], atol=1e-12)


def test_f_sharpens_monotonically():
    """Property (3) of §2.3: with growing s the distance to Q shrinks (away from the
    threshold)."""
    x = np.linspace(-2, 2, 401)
    D = 0.5
    x = x[np.abs(np.abs(x) - D) > 0.05]
    errs = [np.abs(O.transition_f(x, s, D) - O.hard_q(x, D)).max() for s in (5, 10, 20, 40, 80)]
    assert all(a > b for a, b in zip(errs, errs[1:]))


@pytest.mark.parametrize("s,D", [(0.625, 0.5), (15.0, 0.45), (30.0, 0.55)])
def test_f_derivatives_match_finite_differences(s, D):
    x = np.linspace(-2, 2, 81)
    h = 1e-6
    dfdx, dfdD = O.transition_f_grads(x, s, D)
    fd_x = (O.transition_f(x + h, s, D) - O.transition_f(x - h, s, D)) / (2 * h)
    fd_D = (O.transition_f(x, s, D + h) - O.transition_f(x, s, D - h)) / (2 * h)
    scale = max(1.0, np.abs(fd_x).max())
    np.testing.assert_allclose(dfdx, fd_x, atol=1e-6 * scale)
    np.testing.assert_allclose(dfdD, fd_D, atol=1e-6 * scale)


# ----------------------------------------------------------------- Eq. 3 statistics

def test_group_stats_closed_form():
    """Two-valued groups [a]*h + [b]*h: mu0 = (a + b)/2, alpha0 = |a - b|/2, and the TWN
    rule's Delta0 = 0.7 * (|a| + |b|)/2 / alpha0.  Groups are consecutive runs of g in the
    row-major flattening (App. B.2), so a 2 x 8 matrix with g = 4 has 4 groups."""
    W = np.array([[1, 1, 3, 3, -2, -2, -2, -2],
                  [0.5, 0.5, -1.5, -1.5, 4, 4, 8, 8]], dtype=np.float64)
    mu0, alpha0, delta0 = O.group_stats(W, 4, O.THR_TWN07)
    np.testing.assert_allclose(mu0, [2, -2, -0.5, 6])
    np.testing.assert_allclose(alpha0, [1, 0, 1, 2])
    np.testing.assert_allclose(delta0, [0.7 * 2 / 1, 0.5, 0.7 * 1 / 1, 0.7 * 6 / 2])
    _, _, d_half = O.group_stats(W, 4, O.THR_HALF)
    np.testing.assert_allclose(d_half, 0.5)


def test_group_stats_equivariance():
    r = np.random.default_rng(3)
    W = r.standard_normal((6, 64))
    mu0, alpha0, _ = O.group_stats(W, 16)
    mu1, alpha1, _ = O.group_stats(3.0 * W + 0.25, 16)
    np.testing.assert_allclose(mu1, 3.0 * mu0 + 0.25, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(alpha1, 3.0 * alpha0, rtol=1e-13)


# ----------------------------------------------------------------- LM reduces to plain ternarization

def _zero_mean_weight(rows, K, g, seed):
    """Groups of the form [v, -v] with v on a 1/64 grid: the group mean is exactly 0."""
    r = np.random.default_rng(seed)
    v = r.integers(-40, 41, size=(rows * K // g, g // 2)) / 64.0
    return np.concatenate([v, -v], axis=1).reshape(rows, K)


def test_identity_modulation_is_unmodulated_ternarization():
    """At identity factors (d_mu, d_alpha, d_delta) = (0, 1, 1) and mu0 = 0, Eq. 3-4 give
    alpha T = alpha0 Q(W; Delta0 alpha0): LM ternarization of What equals plain threshold
    ternarization of W scaled by alpha0."""
    g = 8
    W = _zero_mean_weight(4, 16, g, 1)
    stats = O.group_stats(W, g, O.THR_HALF)
    assert np.all(stats[0] == 0)
    G = W.size // g
    ident = (np.zeros(G), np.ones(G), np.ones(G))
    Wq, T, _, alpha, _ = O.ternary_weight(W, g, stats, ident, O.PHASE_HARD, 30.0)
    alpha0 = np.repeat(stats[1], g).reshape(W.shape)
    thr = 0.5 * alpha0
    plain = np.where(W > thr, 1.0, np.where(W < -thr, -1.0, 0.0))
    np.testing.assert_array_equal(T, plain)
    np.testing.assert_allclose(Wq, alpha0 * plain, rtol=0, atol=0)


def test_twn_rule_at_identity_factors():
    """With Delta0 from TWN's rule (§2.2) and identity factors the hard codes are TWN's
    Q(W; 0.7 mean|W|) for zero-mean groups (channel-wise groups, one per row)."""
    K = 32
    W = _zero_mean_weight(5, K, K, 2)
    stats = O.group_stats(W, K, O.THR_TWN07)
    G = W.shape[0]
    ident = (np.zeros(G), np.ones(G), np.ones(G))
    _, T, _, _, _ = O.ternary_weight(W, K, stats, ident, O.PHASE_HARD, 30.0)
    thr = 0.7 * np.abs(W).mean(axis=1, keepdims=True)
    twn = np.where(W > thr, 1.0, np.where(W < -thr, -1.0, 0.0))
    np.testing.assert_array_equal(T, twn)


def test_modulation_shifts_and_scales():
    """d_mu shifts the centre by d_mu * alpha0 and d_alpha rescales: for a group with
    mu0 = 0, alpha0 = 1, the element W = mu + alpha * x maps to What = x (Eq. 3)."""
    g = 4
    W = np.array([[1.0, -1.0, 1.0, -1.0]])
    stats = O.group_stats(W, g)
    assert stats[0][0] == 0 and stats[1][0] == 1
    d_mu, d_alpha = 0.25, 2.0
    mu, alpha, Delta = O.modulation(*stats, [d_mu], [d_alpha], [1.5])
    assert mu[0] == 0.25 and alpha[0] == 2.0 and Delta[0] == 0.75
    x = np.array([0.1, -0.3, 1.2, -2.0])
    W2 = (0.25 + 2.0 * x)[None, :]
    What = O.transformed_weight(W2, g, mu, alpha)
    np.testing.assert_allclose(What.reshape(-1), x, rtol=1e-15)


# ----------------------------------------------------------------- forward / loss special cases

def test_teacher_forward_identity_input():
    """Eq. 6 at t = 0 leaves W untouched; with X = I the output is W^T."""
    r = np.random.default_rng(5)
    W = r.standard_normal((6, 8))
    stats = O.group_stats(W, 4)
    G = W.size // 4
    fac = (np.zeros(G), np.ones(G), np.ones(G))
    Wq = O.ternary_weight(W, 4, stats, fac, O.PHASE_TEACHER, 0.0)[0]
    Y = O.linear_fwd(np.eye(8), Wq)
    np.testing.assert_array_equal(Y, W.T)


def test_hard_forward_is_integer_code_gemm_scaled_per_group():
    """With T in {-1,0,1} and integer X, Y = X (alpha T)^T equals, per group of g input
    columns, alpha times the exact integer product X_block T_block^T."""
    r = np.random.default_rng(9)
    N, K, g, M = 6, 16, 4, 5
    W = r.standard_normal((N, K))
    stats = O.group_stats(W, g)
    G = N * K // g
    fac = (r.uniform(-0.1, 0.1, G), r.uniform(0.8, 1.2, G), r.uniform(0.8, 1.2, G))
    Wq, T, _, alpha, _ = O.ternary_weight(W, g, stats, fac, O.PHASE_HARD, 30.0)
    X = r.integers(-5, 6, size=(M, K))
    Ti = T.astype(np.int64)
    a = alpha.reshape(N, K // g)
    Y = np.zeros((M, N))
    for blk in range(K // g):
        cols = slice(blk * g, (blk + 1) * g)
        Y += (X[:, cols] @ Ti[:, cols].T) * a[:, blk][None, :]
    np.testing.assert_allclose(O.linear_fwd(X, Wq), Y, rtol=1e-13, atol=1e-13)


def test_recon_loss_constant_offset():
    Y_ref = np.random.default_rng(1).standard_normal((3, 4))
    loss, dY = O.recon_loss(Y_ref + 0.5, Y_ref, 0)
    assert abs(loss - 0.25) < 1e-15
    np.testing.assert_allclose(dY, np.full((3, 4), 2 * 0.5 / 12))
    loss_s, dY_s = O.recon_loss(Y_ref + 0.5, Y_ref, 1)
    assert abs(loss_s - 0.25 * 12) < 1e-13
    np.testing.assert_allclose(dY_s, 1.0)


# ----------------------------------------------------------------- gradients (finite differences)

def _tiny(seed=0, N=4, K=8, g=4, M=3):
    r = np.random.default_rng(seed)
    W = r.standard_normal((N, K)) * 0.05
    X = r.standard_normal((M, K))
    stats = O.group_stats(W, g)
    G = N * K // g
    fac = [r.uniform(-0.1, 0.1, G), r.uniform(0.8, 1.2, G), r.uniform(0.8, 1.2, G)]
    return W, X, g, stats, fac


def _loss(W, X, g, stats, fac, s, Y_ref):
    Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_SOFT, s)[0]
    return O.recon_loss(O.linear_fwd(X, Wq), Y_ref)[0]


@pytest.mark.parametrize("s", [0.625, 15.0, 30.0])
def test_soft_gradients_match_central_differences(s):
    """Analytic dX and factor gradients of the SOFT step against central differences of
    the oracle's loss (teacher output held fixed), h = 1e-6, relative agreement 1e-6."""
    W, X, g, stats, fac = _tiny()
    Y_ref = O.linear_fwd(X, W)
    Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_SOFT, s)[0]
    _, dY = O.recon_loss(O.linear_fwd(X, Wq), Y_ref)
    dX, gmu, galpha, gdelta = O.linear_bwd(X, dY, W, g, stats, fac, O.PHASE_SOFT, s)
    h = 1e-6
    for which, analytic in ((0, gmu), (1, galpha), (2, gdelta)):
        fd = np.zeros_like(analytic)
        for j in range(analytic.size):
            fp = [a.copy() for a in fac]
            fm = [a.copy() for a in fac]
            fp[which][j] += h
            fm[which][j] -= h
            fd[j] = (_loss(W, X, g, stats, fp, s, Y_ref) - _loss(W, X, g, stats, fm, s, Y_ref)) / (2 * h)
        scale = np.abs(fd).max()
        np.testing.assert_allclose(analytic, fd, atol=1e-6 * scale + 1e-12)
    fdX = np.zeros_like(X)
    for idx in np.ndindex(*X.shape):
        Xp, Xm = X.copy(), X.copy()
        Xp[idx] += h
        Xm[idx] -= h
        lp = O.recon_loss(O.linear_fwd(Xp, Wq), Y_ref)[0]
        lm = O.recon_loss(O.linear_fwd(Xm, Wq), Y_ref)[0]
        fdX[idx] = (lp - lm) / (2 * h)
    np.testing.assert_allclose(dX, fdX, atol=1e-6 * np.abs(fdX).max())


def test_bwd_uses_transposes_correctly_non_square():
    """Shapes of dX [M, K] and G = dY^T X [N, K] on a non-square layer (M != N != K)."""
    W, X, g, stats, fac = _tiny(seed=4, N=6, K=12, g=4, M=5)
    Y_ref = O.linear_fwd(X, W)
    step = O.calibration_step(X, W, g, stats, fac, O.PHASE_SOFT, 15.0)
    assert step["dX"].shape == X.shape and step["Y"].shape == (5, 6)
    assert step["g_dmu"].shape == (6 * 12 // 4,)
    np.testing.assert_allclose(step["Y_ref"], Y_ref)


def _golden(name):
    vals = {}
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", name)) as fh:
        for line in fh:
            if line.startswith("#") or ":" not in line:
                continue
            k, v = line.split(":", 1)
            vals[k.strip()] = np.array([float(t) for t in v.split()])
    return vals


def test_hard_gradients_hand_computed_golden():
    """The HARD-phase reading (§2.3, stage 2 keeps the last soft iteration's gradients) on a
    hand-computed group at s = 2, where f and Q differ (tests/golden/hard_grad_example.txt):
    the alpha term must use the forward value T = Q; substituting T = f moves g_dalpha from
    -0.472 to -0.408 and fails.  The same numbers pin d_mu and d_delta's derivatives of Eq. 5,
    and the SOFT phase must reproduce the T = f value."""
    gd = _golden("hard_grad_example.txt")
    W = gd["W"].reshape(1, 4)
    Gw = gd["G"].reshape(1, 4)
    s = float(gd["s"][0])
    stats = O.group_stats(W, 4)
    fac = (np.zeros(1), np.ones(1), np.ones(1))
    got = O.factor_grads_from_G(Gw, W, 4, stats, fac, O.PHASE_HARD, s)
    for name, v in zip(("g_dmu", "g_dalpha", "g_ddelta"), got):
        np.testing.assert_allclose(v, gd[name], rtol=1e-12, err_msg=name)
    assert abs(got[1][0] - gd["g_dalpha_if_T_were_f"][0]) > 0.05
    soft = O.factor_grads_from_G(Gw, W, 4, stats, fac, O.PHASE_SOFT, s)
    np.testing.assert_allclose(soft[1], gd["g_dalpha_if_T_were_f"], rtol=1e-12)
    np.testing.assert_allclose(soft[0], gd["g_dmu"], rtol=1e-12)
    np.testing.assert_allclose(soft[2], gd["g_ddelta"], rtol=1e-12)


def test_hard_gradients_reading_self_consistency():
    """HARD-phase factor gradients (parity unpinned: §2.3's stage-2 rule read as a
    surrogate) coincide with the SOFT ones at the same large s when no element sits
    near its threshold, where f and Q agree."""
    r = np.random.default_rng(12)
    g = 4
    N, K, M = 4, 8, 6
    x = r.choice([-1.3, -0.9, -0.2, 0.1, 0.8, 1.4], size=(N, K))
    W = x * 0.05
    stats = O.group_stats(W, g)
    G = N * K // g
    fac = [np.zeros(G), np.ones(G), np.ones(G)]
    X = r.standard_normal((M, K))
    dY = r.standard_normal((M, N))
    s = 400.0
    soft = O.linear_bwd(X, dY, W, g, stats, fac, O.PHASE_SOFT, s)
    hard = O.linear_bwd(X, dY, W, g, stats, fac, O.PHASE_HARD, s)
    What = O.transformed_weight(W, g, *O.modulation(*stats, *fac)[:2])
    assert np.abs(np.abs(What) - 0.5).min() > 0.05
    for a, b in zip(soft, hard):
        np.testing.assert_allclose(a, b, rtol=1e-9, atol=1e-12)


def test_teacher_bwd_has_zero_factor_grads():
    W, X, g, stats, fac = _tiny()
    dY = np.ones((X.shape[0], W.shape[0]))
    dX, a, b, c = O.linear_bwd(X, dY, W, g, stats, fac, O.PHASE_TEACHER, 0.0)
    np.testing.assert_allclose(dX, dY @ W)
    assert not a.any() and not b.any() and not c.any()


def test_degenerate_group_is_zero():
    """A constant group has alpha0 = 0: its Wq, hard codes and gradients are 0."""
    W = np.array([[0.3, 0.3, 0.3, 0.3, 1.0, -1.0, 0.5, -0.5]])
    stats = O.group_stats(W, 4)
    assert stats[1][0] == 0
    fac = (np.zeros(2), np.ones(2), np.ones(2))
    Wq, T, _, _, _ = O.ternary_weight(W, 4, stats, fac, O.PHASE_SOFT, 30.0)
    assert not Wq[0, :4].any()
    codes, _, _ = O.hard_codes(W, 4, stats, fac)
    assert not codes[:4].any()
    X = np.ones((2, 8))
    dY = np.ones((2, 1))
    _, gm, ga, gd = O.linear_bwd(X, dY, W, 4, stats, fac, O.PHASE_SOFT, 30.0)
    assert gm[0] == 0 and ga[0] == 0 and gd[0] == 0


# ----------------------------------------------------------------- packing

def _golden_pack():
    codes = bytes_ = None
    with open(os.path.join(GOLDEN, "pack_example.txt")) as fh:
        for line in fh:
            if line.startswith("codes:"):
                codes = [int(v) for v in line.split(":")[1].split()]
            elif line.startswith("bytes:"):
                bytes_ = [int(v) for v in line.split(":")[1].split()]
    return np.array(codes), np.array(bytes_, dtype=np.uint8)


def test_pack_hand_example():
    codes, expect = _golden_pack()
    np.testing.assert_array_equal(O.pack_codes(codes), expect)


def test_pack_round_trip():
    T = np.random.default_rng(2).integers(-1, 2, 4096)
    np.testing.assert_array_equal(O.unpack_codes(O.pack_codes(T), T.size), T)


# ---------------------------------------------------------------- deployed-form inference

def _golden_infer():
    vals = {}
    path = os.path.join(os.path.dirname(__file__), "golden", "ternary_infer_example.txt")
    for line in open(path):
        if line.startswith("#") or ":" not in line:
            continue
        k, v = line.split(":", 1)
        vals[k.strip()] = np.array(v.split(), dtype=np.float64)
    return vals


def test_ternary_infer_hand_example():
    v = _golden_infer()
    X = np.stack([v["x0"], v["x1"]])
    Y = O.ternary_infer(v["bytes"].astype(np.uint8), v["alpha"], 2, 4, 2, X)
    np.testing.assert_array_equal(Y, np.stack([v["y0"], v["y1"]]))


def test_ternary_infer_is_the_hard_forward():
    """Packing a layer's hard codes and inferring from them gives the HARD-phase forward."""
    r = np.random.default_rng(11)
    N, K, g, M = 6, 256, 128, 5
    W = r.standard_normal((N, K)) * 0.02
    X = r.standard_normal((M, K))
    G = N * K // g
    stats = O.group_stats(W, g, O.THR_HALF)
    fac = (r.uniform(-0.1, 0.1, G), r.uniform(0.8, 1.2, G), r.uniform(0.8, 1.2, G))
    T, alpha, _ = O.hard_codes(W, g, stats, fac)
    Y = O.ternary_infer(O.pack_codes(T), alpha, N, K, g, X)
    Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_HARD, 30.0)[0]
    np.testing.assert_allclose(Y, O.linear_fwd(X, Wq), rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- static scale/threshold rules

def test_absmean_and_twn_static_closed_form():
    """§2.2's static approximations on a hand-computed group (g = 4):
    W = [3, -1, 0.5, -0.2]: mean|W| = 1.175.
    absmean: alpha = 1.175, Delta = alpha / 2 (0.5 in What = W / alpha units).
    TWN: Delta_W = 0.7 * 1.175 = 0.8225; elements above it: 3 and -1, alpha = 2,
    Delta0 = 0.8225 / 2 = 0.41125."""
    W = np.array([[3.0, -1.0, 0.5, -0.2]])
    mu0, a0, d0 = O.group_stats(W, 4, O.THR_ABSMEAN)
    np.testing.assert_allclose([mu0[0], a0[0], d0[0]], [0.0, 1.175, 0.5], rtol=0, atol=1e-15)
    mu0, a0, d0 = O.group_stats(W, 4, O.THR_TWN_STATIC)
    np.testing.assert_allclose([mu0[0], a0[0], d0[0]], [0.0, 2.0, 0.41125], rtol=0, atol=1e-15)


def test_static_rules_at_identity_factors_are_the_papers_ternarizations():
    """At identity factors the hard ternarization reproduces each rule as §2.2 states it:
    absmean: T = sign(W) [|W| > mean|W| / 2], alpha = mean|W|;
    TWN: T = sign(W) [|W| > 0.7 mean|W|], alpha = mean |W| over the kept elements."""
    r = np.random.default_rng(12)
    N, K, g = 5, 128, 64
    W = r.standard_normal((N, K)) * 0.02
    G = N * K // g
    ident = (np.zeros(G), np.ones(G), np.ones(G))
    Wg = W.reshape(G, g)
    mean_abs = np.abs(Wg).mean(axis=1)
    for rule, thr, alpha in (
            (O.THR_ABSMEAN, mean_abs / 2, mean_abs),
            (O.THR_TWN_STATIC, 0.7 * mean_abs,
             np.array([np.abs(w[np.abs(w) > 0.7 * m]).mean() for w, m in zip(Wg, mean_abs)]))):
        stats = O.group_stats(W, g, rule)
        T, a, _ = O.hard_codes(W, g, stats, ident)
        want_T = np.sign(Wg) * (np.abs(Wg) > thr[:, None])
        np.testing.assert_array_equal(T.reshape(G, g), want_T)
        np.testing.assert_allclose(a, alpha, rtol=1e-12)


# ---------------------------------------------------------------- W ~ alpha T + mu variant

def test_mu_reconstruction_reproduces_two_valued_groups():
    """A group holding two values a < b is mu0 = (a + b)/2, alpha0 = (b - a)/2, What = -1 / +1
    (Eq. 3), so at identity factors the hard ternarization with mu (tab:mu's variant) gives
    alpha T + mu = W exactly, while without mu it gives -alpha0 / +alpha0."""
    W = np.array([[1.0, 3.0, 3.0, 1.0, -2.0, -1.0, -1.0, -2.0]])
    g = 4
    stats = O.group_stats(W, g)
    ident = (np.zeros(2), np.ones(2), np.ones(2))
    Wq_mu = O.ternary_weight(W, g, stats, ident, O.PHASE_HARD, 30.0, with_mu=True)[0]
    np.testing.assert_array_equal(Wq_mu, W)
    Wq = O.ternary_weight(W, g, stats, ident, O.PHASE_HARD, 30.0)[0]
    np.testing.assert_array_equal(Wq, [[-1, 1, 1, -1, -0.5, 0.5, 0.5, -0.5]])


@pytest.mark.parametrize("s", [0.625, 30.0])
def test_mu_variant_gradients_match_central_differences(s):
    """With mu in the reconstruction the factor gradients (dWq/dmu = 1 - f') still match
    central differences of the loss."""
    W, X, g, stats, fac = _tiny(seed=3)
    Y_ref = O.linear_fwd(X, W)

    def loss(f):
        Wq = O.ternary_weight(W, g, stats, f, O.PHASE_SOFT, s, with_mu=True)[0]
        return O.recon_loss(O.linear_fwd(X, Wq), Y_ref)[0]

    Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_SOFT, s, with_mu=True)[0]
    _, dY = O.recon_loss(O.linear_fwd(X, Wq), Y_ref)
    dX, gmu, galpha, gdelta = O.linear_bwd(X, dY, W, g, stats, fac, O.PHASE_SOFT, s, with_mu=True)
    np.testing.assert_allclose(dX, dY @ Wq)
    h = 1e-6
    for which, analytic in ((0, gmu), (1, galpha), (2, gdelta)):
        fd = np.zeros_like(analytic)
        for j in range(analytic.size):
            fp = [a.copy() for a in fac]
            fm = [a.copy() for a in fac]
            fp[which][j] += h
            fm[which][j] -= h
            fd[j] = (loss(fp) - loss(fm)) / (2 * h)
        np.testing.assert_allclose(analytic, fd, atol=1e-6 * np.abs(fd).max() + 1e-12)


def test_ternary_infer_with_mu_is_the_hard_forward_with_mu():
    r = np.random.default_rng(13)
    N, K, g, M = 4, 128, 64, 3
    W = r.standard_normal((N, K)) * 0.02
    X = r.standard_normal((M, K))
    G = N * K // g
    stats = O.group_stats(W, g)
    fac = (r.uniform(-0.1, 0.1, G), r.uniform(0.8, 1.2, G), r.uniform(0.8, 1.2, G))
    T, alpha, _ = O.hard_codes(W, g, stats, fac)
    mu = O.modulation(*stats, *fac)[0]
    Y = O.ternary_infer(O.pack_codes(T), alpha, N, K, g, X, mu=mu)
    Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_HARD, 30.0, with_mu=True)[0]
    np.testing.assert_allclose(Y, O.linear_fwd(X, Wq), rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- direct learning (Fig. fig:error)

@pytest.mark.parametrize("s", [0.625, 30.0])
def test_direct_learning_is_a_reparametrization_of_the_modulation(s):
    """Learning alpha and a weight-space threshold Delta_W directly (the comparison of
    Fig. fig:error), from a static rule's statistics (mu0 = 0), is the modulation with
    d_mu = 0 under alpha = d_alpha alpha0, Delta_W = alpha d_delta Delta0: the forward is the
    same function, and the direct parameters' gradients follow from the factor gradients by
    the chain rule.  Checked against central differences of the direct parametrisation."""
    W, X, g, _, fac = _tiny(seed=5)
    stats = O.group_stats(W, g, O.THR_ABSMEAN)
    mu0, alpha0, delta0 = stats
    assert not mu0.any()
    G = alpha0.size
    zero = np.zeros(G)
    a_d = fac[1] * alpha0                      # direct scale
    D_d = a_d * fac[2] * delta0                # direct threshold in W units
    Y_ref = O.linear_fwd(X, W)

    def loss_direct(a, D):
        f = (zero, a / alpha0, (D / a) / delta0)
        return O.recon_loss(O.linear_fwd(X, O.ternary_weight(W, g, stats, f, O.PHASE_SOFT, s)[0]), Y_ref)[0]

    f0 = (zero, fac[1], fac[2])
    Wq = O.ternary_weight(W, g, stats, f0, O.PHASE_SOFT, s)[0]
    _, dY = O.recon_loss(O.linear_fwd(X, Wq), Y_ref)
    _, _, g_dalpha, g_ddelta = O.linear_bwd(X, dY, W, g, stats, f0, O.PHASE_SOFT, s)
    want_a = g_dalpha / alpha0 - g_ddelta * D_d / (a_d * a_d * delta0)
    want_D = g_ddelta / (a_d * delta0)
    h = 1e-7
    for which, want in ((0, want_a), (1, want_D)):
        fd = np.zeros(G)
        for j in range(G):
            p = [a_d.copy(), D_d.copy()]
            m = [a_d.copy(), D_d.copy()]
            scale = p[which][j]
            p[which][j] += h * scale
            m[which][j] -= h * scale
            fd[j] = (loss_direct(*p) - loss_direct(*m)) / (2 * h * scale)
        np.testing.assert_allclose(want, fd, rtol=1e-4, atol=1e-6 * np.abs(fd).max())


# ----------------------------------------------------------------- App. B.1: schedule and AdamW update

def test_schedule_at_epoch_paper_defaults():
    """App. B.1 (m = 60, gamma = 0.8, s0 = 30) with §2.3's t = e / m: 48 soft epochs whose
    sharpness rises linearly from s0 / 48 to exactly s0, then 12 hard epochs at s0; t = 0 is
    the teacher."""
    m, gamma, s0 = 60, 0.8, 30.0
    assert O.schedule_at_epoch(0, m, gamma, s0)[0] == O.PHASE_TEACHER
    pts = [O.schedule_at_epoch(e, m, gamma, s0) for e in range(1, m + 1)]
    phases = [p for p, _ in pts]
    assert phases == [O.PHASE_SOFT] * 48 + [O.PHASE_HARD] * 12
    s = np.array([v for _, v in pts[:48]])
    np.testing.assert_allclose(s, 0.625 * np.arange(1, 49), rtol=1e-15)
    assert s[-1] == s0
    assert all(v == s0 for _, v in pts[48:])
    # gamma = 1: no hard stage; gamma m not an integer: floor(gamma m) soft epochs
    assert [O.schedule_at_epoch(e, 10, 1.0, 5.0)[0] for e in range(1, 11)] == [O.PHASE_SOFT] * 10
    assert sum(O.schedule_at_epoch(e, 7, 0.5, 5.0)[0] == O.PHASE_SOFT for e in range(1, 8)) == 3
    # rounding of gamma m (0.57 * 100 = 56.99999999999999 in fp64) does not drop an epoch
    assert sum(O.schedule_at_epoch(e, 100, 0.57, 5.0)[0] == O.PHASE_SOFT for e in range(1, 101)) == 57


def test_hard_stage_keeps_the_last_soft_sharpness():
    """§2.3: the hard stage takes the gradients of the first stage's last iteration, so its
    backward sharpness is the last soft epoch's.  With gamma m = 7.5 (m = 10, gamma = 0.75)
    the soft stage ends at e = 7 with s = (0.7 / 0.75) s0 = 28 for s0 = 30, not s0; with
    gamma m < 1 there is no soft epoch and s0 is kept."""
    m, gamma, s0 = 10, 0.75, 30.0
    phases = [O.schedule_at_epoch(e, m, gamma, s0) for e in range(1, m + 1)]
    assert [p for p, _ in phases] == [O.PHASE_SOFT] * 7 + [O.PHASE_HARD] * 3
    last_soft = phases[6][1]
    assert last_soft == pytest.approx(28.0, rel=1e-15)
    assert all(s == last_soft for _, s in phases[7:])
    assert [O.schedule_at_epoch(e, 3, 0.2, s0) for e in (1, 2, 3)] == [(O.PHASE_HARD, s0)] * 3


def test_linear_decay_lr_closed_form():
    """A linear decay to zero: lr0 at the first update, equal decrements lr0 / total, the
    last update at lr0 / total, and the sum lr0 (total + 1) / 2."""
    lr0, total = 1e-3, 171
    lrs = np.array([O.linear_decay_lr(lr0, k, total) for k in range(total)])
    assert lrs[0] == lr0
    np.testing.assert_allclose(np.diff(lrs), -lr0 / total, rtol=1e-9)
    np.testing.assert_allclose(lrs[-1], lr0 / total, rtol=1e-12)
    np.testing.assert_allclose(lrs.sum(), lr0 * (total + 1) / 2, rtol=1e-12)


def test_adamw_first_step_and_constant_gradient_closed_forms():
    """From zero moments the bias correction makes m_hat = g and v_hat = g^2 exactly, so the
    first step is p (1 - lr wd) - lr g / (|g| + eps); under a constant gradient the same
    holds at every step (m_t = g (1 - beta1^t)), so each step moves p by lr g / (|g| + eps)."""
    r = np.random.default_rng(3)
    p0 = r.uniform(-1, 1, 64)
    g = r.normal(0, 1e-3, 64)
    z = np.zeros(64)
    lr, wd, eps = 1e-3, 0.01, 1e-8
    p1, m1, v1 = O.adamw_step(p0, g, z, z, 1, lr, 0.9, 0.999, eps, wd)
    np.testing.assert_allclose(p1, p0 * (1 - lr * wd) - lr * g / (np.abs(g) + eps), rtol=1e-13, atol=1e-18)
    np.testing.assert_allclose(m1, 0.1 * g, rtol=1e-13)
    np.testing.assert_allclose(v1, 0.001 * g * g, rtol=1e-12)
    p, m, v = p0, z, z
    lrs = [1e-3 * (1 - k / 10) for k in range(10)]
    for t, lr_t in enumerate(lrs, start=1):
        p, m, v = O.adamw_step(p, g, m, v, t, lr_t, 0.8, 0.95, eps, 0.0)
    np.testing.assert_allclose(p, p0 - sum(lrs) * g / (np.abs(g) + eps), rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("betas,eps,wd", [((0.9, 0.999), 1e-8, 0.0), ((0.9, 0.999), 1e-8, 0.01),
                                          ((0.8, 0.95), 1e-6, 0.1)])
def test_adamw_matches_torch_adamw(betas, eps, wd):
    """Eight updates with a decaying learning rate and changing gradients against PyTorch's
    own AdamW (fp64 on the CPU, single-tensor path): parameters and both moments."""
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(11)
    p0 = r.uniform(0.5, 1.5, 257)
    grads = [r.normal(0, 10.0 ** -r.integers(2, 6), 257) for _ in range(8)]
    param = torch.nn.Parameter(torch.from_numpy(p0.copy()))
    opt = torch.optim.AdamW([param], lr=1e-3, betas=betas, eps=eps, weight_decay=wd, foreach=False)
    p, m, v = p0, np.zeros(257), np.zeros(257)
    for k, gk in enumerate(grads):
        lr = 1e-3 * (1 - k / 8)
        for grp in opt.param_groups:
            grp["lr"] = lr
        param.grad = torch.from_numpy(gk.copy())
        opt.step()
        p, m, v = O.adamw_step(p, gk, m, v, k + 1, lr, betas[0], betas[1], eps, wd)
    state = opt.state[param]
    np.testing.assert_allclose(p, param.detach().numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(m, state["exp_avg"].numpy(), rtol=1e-12, atol=1e-20)
    np.testing.assert_allclose(v, state["exp_avg_sq"].numpy(), rtol=1e-12, atol=1e-30)


def test_factor_update_projects_onto_the_constraints():
    """§2.2's constraints after the update: values inside the sets are untouched, values
    outside land on the nearest bound, NaN stays NaN; each factor uses its own gradient and
    its own moments."""
    margin = 1e-4
    mu, al, de = O.project_factors([-1.5, -0.5, 0.99995, np.nan], [-2.0, 0.0, 0.5, 3.0], [1e-5, 2.0, -1.0, 0.2],
                                   margin)
    np.testing.assert_array_equal(mu[:3], [-1 + margin, -0.5, 1 - margin])
    assert np.isnan(mu[3])
    np.testing.assert_array_equal(al, [margin, margin, 0.5, 3.0])
    np.testing.assert_array_equal(de, [margin, 2.0, margin, 0.2])
    # gradients routed to their own factor: only d_alpha moves when only its gradient is set
    f = (np.zeros(4), np.ones(4), np.ones(4))
    gr = (np.zeros(4), np.full(4, 0.3), np.zeros(4))
    (nm, na, nd), mom = O.factor_update(f, gr, (np.zeros(4),) * 6, 1, 1e-3)
    np.testing.assert_array_equal(nm, 0.0)
    np.testing.assert_array_equal(nd, 1.0)
    np.testing.assert_allclose(na, 1.0 - 1e-3 * 0.3 / (0.3 + 1e-8), rtol=1e-14)
    np.testing.assert_allclose(mom[1], 0.1 * 0.3, rtol=1e-14)
    np.testing.assert_allclose(mom[4], 0.001 * 0.09, rtol=1e-13)


def test_calibration_loop_lowers_the_hard_reconstruction_error():
    """The pieces compose into App. B.1's calibration: 60 epochs of three batches at the
    paper's schedule (gamma = 0.8, s0 = 30) and optimizer (AdamW, 1e-3 decayed linearly to
    zero), each step's gradients driving the update, end with factors whose hard-ternarized
    layer reconstructs the teacher better than the static initialization does (seeded tiny
    layer; the loop reaches 0.82 of the initial loss, the bound leaves a margin)."""
    r = np.random.default_rng(0)
    N, K, g, M = 16, 64, 16, 96
    W = r.standard_normal((N, K)) * 0.02
    X = r.standard_normal((M, K))
    stats = O.group_stats(W, g)
    G = N * K // g
    fac, mom = (np.zeros(G), np.ones(G), np.ones(G)), (np.zeros(G),) * 6

    def hard_loss(f):
        return O.calibration_step(X, W, g, stats, f, O.PHASE_HARD, 30.0)["loss"]

    start = hard_loss(fac)
    m, batches, t = 60, 3, 0
    for e in range(1, m + 1):
        phase, s = O.schedule_at_epoch(e, m, 0.8, 30.0)
        for b in range(batches):
            step = O.calibration_step(X[b::batches], W, g, stats, fac, phase, s)
            lr = O.linear_decay_lr(1e-3, t, m * batches)
            t += 1
            fac, mom = O.factor_update(fac, (step["g_dmu"], step["g_dalpha"], step["g_ddelta"]), mom, t, lr)
    assert hard_loss(fac) < 0.9 * start


# ----------------------------------------------------------------- W1.58A8: 8-bit activations

def test_act_quant_a8_exact_on_its_own_grid():
    """Rows that already lie on an 8-bit grid whose largest entry is +-127 steps come back
    exactly: the scale is the grid step (a power of two here, so fp32 division is exact)
    and the codes are the integers; each row has its own scale (per token)."""
    r = np.random.default_rng(30)
    M, K = 5, 48
    steps = 2.0 ** r.integers(-12, -2, M)
    ints = r.integers(-127, 128, (M, K))
    ints[np.arange(M), r.integers(0, K, M)] = np.where(r.random(M) < 0.5, 127, -127)
    X = ints * steps[:, None]
    q, scale = O.act_quant_a8(X)
    np.testing.assert_array_equal(scale, steps.astype(np.float32))
    np.testing.assert_array_equal(q, ints)


def test_act_quant_a8_error_bound_and_range():
    """Round-to-nearest on a symmetric grid: every element within half a step of scale q,
    codes in [-127, 127], the row's absmax at +-127, and a zero row giving zero codes."""
    r = np.random.default_rng(31)
    X = (r.standard_t(4.0, (64, 200)) * 3).astype(np.float32)
    X[7] = 0.0
    q, scale = O.act_quant_a8(X)
    assert np.abs(q).max() <= 127
    err = np.abs(X.astype(np.float64) - q * scale[:, None].astype(np.float64))
    assert np.all(err <= 0.5 * scale[:, None] * (1 + 1e-6) + 1e-30)
    live = np.arange(64) != 7
    assert np.all(np.abs(q[live]).max(axis=1) == 127)
    assert scale[7] == 0 and not q[7].any()


def test_act_quant_a8_is_the_nearest_code_by_brute_force():
    """Each code is the integer in [-127, 127] nearest to x / scale (all 255 candidates
    tried; ties, if any, to the even one)."""
    r = np.random.default_rng(32)
    X = r.standard_normal((6, 40)).astype(np.float32)
    q, scale = O.act_quant_a8(X)
    cand = np.arange(-127, 128)
    for m in range(6):
        u = X[m].astype(np.float32) / scale[m]
        dist = np.abs(u[:, None].astype(np.float64) - cand[None, :])
        best = dist.min(axis=1)
        np.testing.assert_allclose(np.abs(u - q[m]), best, atol=1e-6)


def test_a8_step_reduces_to_the_plain_step_on_grid_inputs():
    """When X already lies on its 8-bit grid the quantizer is the identity, so the A8 step
    (teacher from X, forward and dW from X_q) equals the plain calibration step."""
    W, X, g, stats, fac = _tiny(seed=33, N=8, K=16, g=8, M=6)
    r = np.random.default_rng(33)
    ints = r.integers(-127, 128, X.shape)
    ints[:, 0] = 127
    X = ints * 2.0 ** -7
    a8 = O.a8_calibration_step(X, W, g, stats, fac, O.PHASE_SOFT, 15.0)
    ref = O.calibration_step(X, W, g, stats, fac, O.PHASE_SOFT, 15.0)
    for k in ("Y", "Y_ref", "dY", "dX", "g_dmu", "g_dalpha", "g_ddelta"):
        np.testing.assert_allclose(a8[k], ref[k], rtol=1e-13, atol=1e-15, err_msg=k)
    assert a8["loss"] == pytest.approx(ref["loss"], rel=1e-13)


# ----------------------------------------------------------------- direct learning (Fig. fig:error)

def test_direct_grads_match_central_differences_of_the_direct_parametrization():
    """DL's gradients in (a, d) = (alpha / alpha0, Delta_W / (alpha0 Delta0)) against central
    differences of the loss written directly in a and d (mu at mu0 = 0 for the absmean rule),
    in the soft phase where the loss is smooth."""
    r = np.random.default_rng(70)
    N, K, g, M = 3, 8, 4, 5
    W = r.standard_normal((N, K)) * 0.05
    X = r.standard_normal((M, K))
    stats = O.group_stats(W, g, O.THR_ABSMEAN)
    G = N * K // g
    a = r.uniform(0.8, 1.2, G)
    d = r.uniform(0.3, 0.7, G)
    s = 8.0
    Y_ref = O.linear_fwd(X, W)

    def loss(a, d):
        fac = (np.zeros(G), a, d / a)
        Wq = O.ternary_weight(W, g, stats, fac, O.PHASE_SOFT, s)[0]
        return O.recon_loss(O.linear_fwd(X, Wq), Y_ref)[0]

    step = O.calibration_step(X, W, g, stats, (np.zeros(G), a, d / a), O.PHASE_SOFT, s)
    ga, gd = O.direct_grads(a, d / a, step["g_dalpha"], step["g_ddelta"])
    h = 1e-6
    for j in range(G):
        e = np.zeros(G)
        e[j] = h
        fa = (loss(a + e, d) - loss(a - e, d)) / (2 * h)
        fd = (loss(a, d + e) - loss(a, d - e)) / (2 * h)
        assert ga[j] == pytest.approx(fa, rel=1e-5, abs=1e-9)
        assert gd[j] == pytest.approx(fd, rel=1e-5, abs=1e-9)


def test_direct_update_is_adamw_on_a_and_d():
    """The update against PyTorch's own AdamW on parameters (a, d) fed the converted
    gradients (fp64, several updates), then the return to (d_alpha, d_delta)."""
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(71)
    G = 64
    dal = r.uniform(0.8, 1.2, G)
    ddl = r.uniform(0.8, 1.2, G)
    ta = torch.tensor(dal.copy(), dtype=torch.float64, requires_grad=True)
    td = torch.tensor(dal * ddl, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([ta, td], lr=1e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.01)
    mom = (np.zeros(G),) * 4
    for t in range(1, 6):
        gal = r.standard_normal(G) * 1e-3
        gdl = r.standard_normal(G) * 1e-3
        ga, gd = O.direct_grads(dal, ddl, gal, gdl)
        ta.grad = torch.tensor(ga)
        td.grad = torch.tensor(gd)
        opt.step()
        dal, ddl, mom = O.direct_update(dal, ddl, gal, gdl, mom, t, 1e-3, weight_decay=0.01, margin=0.0)
        np.testing.assert_allclose(dal, ta.detach().numpy(), rtol=1e-13)
        np.testing.assert_allclose(dal * ddl, td.detach().numpy(), rtol=1e-13)


def test_group_recon_error_closed_form():
    """A group [v, -v, 3v, -3v] under absmean (alpha = 2|v|, Delta = |v|): Q gives 0, 0, 1, -1,
    so the error is (v^2 + v^2 + v^2 + v^2) / 4 = v^2 (v a power of two: every value is exact,
    and the two small elements sit exactly on the threshold, where Eq. 2 gives 0)."""
    v = 2.0 ** -7
    W = np.array([[v, -v, 3 * v, -3 * v]])
    stats = O.group_stats(W, 4, O.THR_ABSMEAN)
    fac = (np.zeros(1), np.ones(1), np.ones(1))
    assert O.group_recon_error(W, 4, stats, fac)[0] == pytest.approx(v * v, rel=1e-12)


# ----------------------------------------------------------------- one decoder block (§2.4, Eq. 7)

def _tiny_block(seed=80, B=2, S=5, nh=4, nkv=2, d=4, I=12, g=4):
    r = np.random.default_rng(seed)
    H = nh * d
    shapes = {"q_proj": (nh * d, H), "k_proj": (nkv * d, H), "v_proj": (nkv * d, H), "o_proj": (H, nh * d),
              "gate_proj": (I, H), "up_proj": (I, H), "down_proj": (H, I)}
    W = {n: r.standard_normal(sh) * 0.3 for n, sh in shapes.items()}
    stats = {n: O.group_stats(W[n], g) for n in shapes}
    fac = {n: (r.uniform(-0.1, 0.1, W[n].size // g), r.uniform(0.8, 1.2, W[n].size // g),
               r.uniform(0.8, 1.2, W[n].size // g)) for n in shapes}
    x = r.standard_normal((B * S, H))
    gamma1 = r.uniform(0.5, 1.5, H)
    gamma2 = r.uniform(0.5, 1.5, H)
    qk = dict(q_norm=r.uniform(0.5, 1.5, d), k_norm=r.uniform(0.5, 1.5, d))
    return dict(x=x, W=W, g=g, stats=stats, fac=fac, gamma1=gamma1, gamma2=gamma2, B=B, S=S, nh=nh, nkv=nkv,
                d=d, base=10000.0, eps=1e-5, qk=qk)


def _block_loss(blk, fac, s, qk_norm=False):
    return O.block_calibration_step(blk["x"], blk["W"], blk["g"], blk["stats"], fac, blk["gamma1"], blk["gamma2"],
                                    blk["B"], blk["S"], blk["nh"], blk["nkv"], blk["d"], blk["base"], blk["eps"],
                                    O.PHASE_SOFT, s, **(blk["qk"] if qk_norm else {}))["loss"]


@pytest.mark.parametrize("qk_norm", [False, True])
def test_block_factor_gradients_match_central_differences(qk_norm):
    """The block's backward (SwiGLU, RMSNorm with the residual, attention with grouped heads,
    rotary embedding, every linear's chain rule; with qk_norm the per-head query/key RMSNorm of
    the Qwen3 block) against central differences of the block loss, for sampled groups of
    every linear and all three factors, soft phase."""
    blk = _tiny_block()
    s = 3.0
    step = O.block_calibration_step(blk["x"], blk["W"], blk["g"], blk["stats"], blk["fac"], blk["gamma1"],
                                    blk["gamma2"], blk["B"], blk["S"], blk["nh"], blk["nkv"], blk["d"], blk["base"],
                                    blk["eps"], O.PHASE_SOFT, s, **(blk["qk"] if qk_norm else {}))
    r = np.random.default_rng(81)
    h = 1e-6
    for name in O.BLOCK_LINEARS:
        G = blk["W"][name].size // blk["g"]
        for q in range(3):
            for j in r.choice(G, 2, replace=False):
                fp = {n: tuple(a.copy() for a in f) for n, f in blk["fac"].items()}
                fm = {n: tuple(a.copy() for a in f) for n, f in blk["fac"].items()}
                fp[name][q][j] += h
                fm[name][q][j] -= h
                fd = (_block_loss(blk, fp, s, qk_norm) - _block_loss(blk, fm, s, qk_norm)) / (2 * h)
                got = step["g"][name][q][j]
                assert got == pytest.approx(fd, rel=1e-5, abs=1e-10 * max(1.0, abs(fd))), (name, q, j)


def test_block_teacher_reconstructs_itself():
    """With the teacher's weights (TEACHER phase) the block output equals the teacher output
    and the loss is zero."""
    blk = _tiny_block(seed=82)
    st = O.block_calibration_step(blk["x"], blk["W"], blk["g"], blk["stats"], blk["fac"], blk["gamma1"],
                                  blk["gamma2"], blk["B"], blk["S"], blk["nh"], blk["nkv"], blk["d"], blk["base"],
                                  blk["eps"], O.PHASE_TEACHER, 0.0)
    np.testing.assert_array_equal(st["out"], st["out_ref"])
    assert st["loss"] == 0.0


def test_attention_closed_forms():
    """Causal attention with all-zero queries gives equal weights to the keys up to each
    query: O at position s is the mean of V over positions 0..s; a single position returns
    its value row; the query head h reads key/value head h // (nh / nkv)."""
    r = np.random.default_rng(83)
    B, S, nh, nkv, d = 2, 6, 4, 2, 3
    v = r.standard_normal((B * S, nkv * d))
    k = r.standard_normal((B * S, nkv * d))
    o, _ = O.attention(np.zeros((B * S, nh * d)), k, v, B, S, nh, nkv, d)
    vb = v.reshape(B, S, nkv, d)
    want = np.cumsum(vb, axis=1) / np.arange(1, S + 1)[None, :, None, None]
    want = np.repeat(want, nh // nkv, axis=2).reshape(B * S, nh * d)
    np.testing.assert_allclose(o, want, rtol=1e-13)
    o1, _ = O.attention(r.standard_normal((B, nh * d)), k[:B], v[:B], B, 1, nh, nkv, d)
    np.testing.assert_allclose(o1, np.repeat(v[:B].reshape(B, nkv, d), nh // nkv, axis=1).reshape(B, nh * d),
                               rtol=1e-13)


def test_attention_gradients_match_central_differences():
    """attention_bwd against central differences of sum(dO * O) in q, k and v."""
    r = np.random.default_rng(84)
    B, S, nh, nkv, d = 1, 4, 2, 1, 4
    q, k, v = (r.standard_normal((B * S, n * d)) for n in (nh, nkv, nkv))
    do = r.standard_normal((B * S, nh * d))
    _, p = O.attention(q, k, v, B, S, nh, nkv, d)
    dq, dk, dv = O.attention_bwd(q, k, v, p, do, B, S, nh, nkv, d)
    f = lambda q, k, v: float((O.attention(q, k, v, B, S, nh, nkv, d)[0] * do).sum())  # noqa: E731
    h = 1e-6
    for arr, grad, which in ((q, dq, 0), (k, dk, 1), (v, dv, 2)):
        for idx in [(0, 0), (S - 1, arr.shape[1] - 1), (1, 2)]:
            args_p = [q.copy(), k.copy(), v.copy()]
            args_m = [q.copy(), k.copy(), v.copy()]
            args_p[which][idx] += h
            args_m[which][idx] -= h
            fd = (f(*args_p) - f(*args_m)) / (2 * h)
            assert grad[idx] == pytest.approx(fd, rel=1e-6, abs=1e-9)


def test_rope_identity_norm_and_inverse():
    """Position 0 is not rotated; every rotated pair keeps its length; the inverse rotation
    undoes the rotation; with d = 2 the angle of position s is exactly s (base^0 = 1)."""
    r = np.random.default_rng(85)
    S, nh, d = 7, 3, 8
    x = r.standard_normal((2 * S, nh * d))
    y = O.rope(x, S, nh, d, 10000.0)
    np.testing.assert_allclose(y[0], x[0], rtol=1e-15)
    xh, yh = x.reshape(-1, nh, d), y.reshape(-1, nh, d)
    nx = xh[..., : d // 2] ** 2 + xh[..., d // 2:] ** 2
    ny = yh[..., : d // 2] ** 2 + yh[..., d // 2:] ** 2
    np.testing.assert_allclose(ny, nx, rtol=1e-12)
    np.testing.assert_allclose(O.rope(y, S, nh, d, 10000.0, inverse=True), x, rtol=1e-12, atol=1e-14)
    z = np.array([[1.0, 0.0]] * 4)
    rz = O.rope(z, 4, 1, 2, 10000.0)
    np.testing.assert_allclose(rz, np.stack([np.cos(np.arange(4.0) % 4), np.sin(np.arange(4.0) % 4)], 1),
                               rtol=1e-15)


def test_rmsnorm_closed_forms():
    """A constant row c maps to gamma * c / sqrt(c^2 + eps); without eps the norm is scale
    invariant; its gradient matches central differences."""
    gamma = np.array([0.5, 2.0, 1.5])
    y, _ = O.rmsnorm(np.full((1, 3), 3.0), gamma, 1e-5)
    np.testing.assert_allclose(y[0], gamma * 3.0 / np.sqrt(9.0 + 1e-5), rtol=1e-15)
    x = np.random.default_rng(86).standard_normal((4, 3))
    np.testing.assert_allclose(O.rmsnorm(7.0 * x, gamma, 0.0)[0], O.rmsnorm(x, gamma, 0.0)[0], rtol=1e-13)
    dy = np.random.default_rng(87).standard_normal((4, 3))
    _, rr = O.rmsnorm(x, gamma, 1e-5)
    dx = O.rmsnorm_bwd(x, gamma, rr, dy)
    h = 1e-6
    for i, j in ((0, 0), (3, 2), (2, 1)):
        xp, xm = x.copy(), x.copy()
        xp[i, j] += h
        xm[i, j] -= h
        fd = ((O.rmsnorm(xp, gamma, 1e-5)[0] - O.rmsnorm(xm, gamma, 1e-5)[0]) * dy).sum() / (2 * h)
        assert dx[i, j] == pytest.approx(fd, rel=1e-6)


def test_attention_logsumexp_closed_form_and_softmax():
    """With q = 0 every allowed score is 0, so query s's normaliser is log(s + 1); on random
    inputs exp(score - lse) over the allowed keys must be ``attention``'s probabilities."""
    B, S, nh, nkv, d = 2, 7, 4, 2, 8
    r = np.random.default_rng(81)
    k = r.standard_normal((B * S, nkv * d))
    lse0 = O.attention_logsumexp(np.zeros((B * S, nh * d)), k, B, S, nh, nkv, d)
    np.testing.assert_allclose(lse0, np.broadcast_to(np.log(np.arange(1, S + 1)), (B, nh, S)), rtol=0, atol=1e-14)
    q = r.standard_normal((B * S, nh * d))
    lse = O.attention_logsumexp(q, k, B, S, nh, nkv, d)
    v = r.standard_normal((B * S, nkv * d))
    _, p = O.attention(q, k, v, B, S, nh, nkv, d)
    qh = q.reshape(B, S, nh, d)
    kh = np.repeat(k.reshape(B, S, nkv, d), nh // nkv, axis=2)
    for b, h, i, j in [(0, 0, 3, 1), (1, 3, 6, 6), (1, 2, 0, 0), (0, 1, 5, 2)]:
        score = qh[b, i, h] @ kh[b, j, h] / np.sqrt(d)
        assert abs(np.exp(score - lse[b, h, i]) - p[b, h, i, j]) < 1e-14
    assert np.all(p[0, 0][np.triu_indices(S, 1)] == 0.0)


def test_swiglu_gradients_match_central_differences():
    r = np.random.default_rng(82)
    gt, u, dm = (r.standard_normal((3, 5)) * 2.0 for _ in range(3))
    d_gt, d_u = O.swiglu_bwd(gt, u, dm)
    h = 1e-6
    num_gt = (np.sum(dm * O.swiglu(gt + h, u)) - np.sum(dm * O.swiglu(gt - h, u))) / (2 * h)
    num_u = (np.sum(dm * O.swiglu(gt, u + h)) - np.sum(dm * O.swiglu(gt, u - h))) / (2 * h)
    # the elementwise map: perturbing everything at once sums the elementwise derivatives
    assert abs(num_gt - d_gt.sum()) < 1e-7 * max(1.0, abs(num_gt))
    assert abs(num_u - d_u.sum()) < 1e-7 * max(1.0, abs(num_u))
    e = np.zeros_like(gt)
    e[1, 2] = h
    one = (np.sum(dm * O.swiglu(gt + e, u)) - np.sum(dm * O.swiglu(gt - e, u))) / (2 * h)
    assert abs(one - d_gt[1, 2]) < 1e-7 * max(1.0, abs(one))
    # silu(0) = 0 and silu's slope at 0 is 1/2
    np.testing.assert_allclose(O.swiglu(np.zeros(2), np.ones(2)), 0.0, atol=0)
    np.testing.assert_allclose(O.swiglu_bwd(np.zeros(1), np.ones(1), np.ones(1))[0], 0.5, rtol=1e-15)


def test_block_head_norm_is_rmsnorm_per_head_and_changes_the_block():
    """The Qwen3 query/key norm normalises each head on its own: scaling one head's q_proj rows
    leaves the block output unchanged (RMSNorm is scale-invariant per row up to eps), while the
    block without the norm changes."""
    blk = _tiny_block(seed=84)
    W2 = {n: w.copy() for n, w in blk["W"].items()}
    W2["q_proj"][: blk["d"]] *= 7.0  # head 0's rows
    args = (blk["gamma1"], blk["gamma2"], blk["B"], blk["S"], blk["nh"], blk["nkv"], blk["d"], blk["base"], 0.0)
    o1, _ = O.block_forward(blk["x"], blk["W"], *args, **blk["qk"])
    o2, _ = O.block_forward(blk["x"], W2, *args, **blk["qk"])
    np.testing.assert_allclose(o1, o2, rtol=1e-12, atol=1e-12)
    p1, _ = O.block_forward(blk["x"], blk["W"], *args)
    p2, _ = O.block_forward(blk["x"], W2, *args)
    assert np.abs(p1 - p2).max() > 1e-3
