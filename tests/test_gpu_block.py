"""GPU vs oracle parity of the decoder-block window (Eq. 7 over one block, §2.4): the layers
between the linears (RMSNorm forward and backward, rotary embedding and its inverse, SwiGLU
forward and backward, the block output with its loss, causal grouped-query attention forward
and backward), each against the oracle's function on the same seeded inputs, then the whole
block calibration step (teacher block, student block at the schedule point, loss, and the
factor gradients of all seven linears through the block's backward) against the oracle's
``block_calibration_step``.

Tolerances: bf16 activations, so the bf16 bar (relative Frobenius error 2e-2) on every
tensor; fp32-only quantities (the residual sum, the RMS factors, the log-sum-exp) against
their fp32 rounding.  Attention is also checked at the Llama-3-8B block's full size (4 x 2048
tokens, 32 query heads, 8 key/value heads, d = 128) on one sampled sequence and key/value
head, all of whose rows the oracle computes."""
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


def _bf16(r, shape, scale=1.0):
    return syn.round_bf16((r.standard_normal(shape) * scale).astype(np.float32))


def _f32(t):
    return U.to_host(t).astype(np.float64)


# ---------------------------------------------------------------- the layers one by one

@pytest.mark.parametrize("T,H,x_dtype", [(300, 512, "bf16"), (7, 4096, "f32"), (1, 136, "bf16"), (1999, 128, "bf16"),
                                         (5, 1032, "f32")])
def test_rmsnorm_fwd_with_residual(device, T, H, x_dtype):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(90, f"rms/{T}/{H}")
    x = _bf16(r, (T, H)) if x_dtype == "bf16" else r.standard_normal((T, H)).astype(np.float32)
    res = _bf16(r, (T, H), 0.5)
    gamma = r.uniform(0.5, 1.5, H).astype(np.float32)
    xd = U.to_device(x, x_dtype, device)
    Z = torch.empty(T, H, dtype=torch.bfloat16, device=device)
    h = torch.empty(T, H, dtype=torch.float32, device=device)
    rr = torch.empty(T, dtype=torch.float32, device=device)
    gd = torch.from_numpy(gamma).to(device)
    C.catq_rmsnorm_fwd(xd, gd, Z, rr, 1e-5, residual=U.to_device(res, "bf16", device), h_out=h)
    hx = x.astype(np.float64) + res.astype(np.float64)
    assert U.max_rel(_f32(h), hx) <= 1e-7
    z_ref, r_ref = O.rmsnorm(hx, gamma, 1e-5)
    assert U.max_rel(_f32(rr), r_ref) <= U.TOL_F32
    assert U.fro_rel(_f32(Z), z_ref) <= U.TOL_BF16
    # without the residual: the plain norm of x
    C.catq_rmsnorm_fwd(xd, gd, Z, rr, 1e-5)
    z0, r0 = O.rmsnorm(x, gamma, 1e-5)
    assert U.max_rel(_f32(rr), r0) <= U.TOL_F32
    assert U.fro_rel(_f32(Z), z0) <= U.TOL_BF16


@pytest.mark.parametrize("h_dtype,H", [("f32", 1024), ("bf16", 1024), ("f32", 2048), ("bf16", 128)])
def test_rmsnorm_bwd_two_consumers_and_residual(device, h_dtype, H):
    """Rows up to 1024 take the warp-per-row kernel, longer ones the CTA-per-row kernel."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    T = 257
    r = syn.rng(91, f"rms_bwd/{h_dtype}/{H}")
    h = r.standard_normal((T, H)).astype(np.float32)
    if h_dtype == "bf16":
        h = syn.round_bf16(h)
    gamma = r.uniform(0.5, 1.5, H).astype(np.float32)
    dz, dz2, dres = _bf16(r, (T, H)), _bf16(r, (T, H)), _bf16(r, (T, H))
    _, r_ref = O.rmsnorm(h, gamma, 1e-5)
    hd = U.to_device(h, h_dtype, device)
    rr = torch.from_numpy(r_ref.astype(np.float32)).to(device)
    gd = torch.from_numpy(gamma).to(device)
    dX = torch.empty(T, H, dtype=torch.bfloat16, device=device)
    C.catq_rmsnorm_bwd(hd, gd, rr, U.to_device(dz, "bf16", device), dX, dZ2=U.to_device(dz2, "bf16", device),
                       d_residual=U.to_device(dres, "bf16", device))
    want = O.rmsnorm_bwd(h, gamma, r_ref.astype(np.float32), dz.astype(np.float64) + dz2) + dres
    assert U.fro_rel(_f32(dX), want) <= U.TOL_BF16
    C.catq_rmsnorm_bwd(hd, gd, rr, U.to_device(dz, "bf16", device), dX)
    assert U.fro_rel(_f32(dX), O.rmsnorm_bwd(h, gamma, r_ref.astype(np.float32), dz)) <= U.TOL_BF16


@pytest.mark.parametrize("S,nh,d,base", [(2048, 8, 128, 500000.0), (5, 3, 64, 10000.0), (7, 2, 24, 10000.0)])
def test_rope_and_inverse(device, S, nh, d, base):
    from paper_2606_26650_gb300 import catq as C
    T = 2 * S
    r = syn.rng(92, f"rope/{S}")
    x = _bf16(r, (T, nh * d))
    xd = U.to_device(x, "bf16", device)
    C.catq_rope(xd, S, nh, d, base)
    assert U.fro_rel(_f32(xd), O.rope(x, S, nh, d, base)) <= U.TOL_BF16
    y = syn.round_bf16(U.to_host(xd))
    C.catq_rope(xd, S, nh, d, base, inverse=True)
    assert U.fro_rel(_f32(xd), O.rope(y, S, nh, d, base, inverse=True)) <= U.TOL_BF16


def test_swiglu_fwd_bwd(device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    r = syn.rng(93, "swiglu")
    n = 1000 * 17 + 5  # not a multiple of the vector width
    gt, u, dm = _bf16(r, n, 2.0), _bf16(r, n), _bf16(r, n)
    gd, ud, dmd = (U.to_device(a, "bf16", device) for a in (gt, u, dm))
    M = torch.empty(n, dtype=torch.bfloat16, device=device)
    C.catq_swiglu_fwd(gd, ud, M)
    assert U.fro_rel(_f32(M), O.swiglu(gt, u)) <= U.TOL_BF16
    dg, du = torch.empty_like(M), torch.empty_like(M)
    C.catq_swiglu_bwd(gd, ud, dmd, dg, du)
    want_g, want_u = O.swiglu_bwd(gt, u, dm)
    assert U.fro_rel(_f32(dg), want_g) <= U.TOL_BF16
    assert U.fro_rel(_f32(du), want_u) <= U.TOL_BF16


@pytest.mark.parametrize("reduction", [0, 1])
def test_block_output_loss(device, reduction):
    """out = h + branch in fp32, the loss on it against an fp32 teacher output and d_out; the
    student-teacher difference is 1e-3 of the residual's size, which a bf16 out would lose."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    T, H = 333, 512
    r = syn.rng(94, "block_loss")
    h = (r.standard_normal((T, H)) * 4.0).astype(np.float32)
    branch = _bf16(r, (T, H), 0.1)
    ref = (h.astype(np.float64) + branch + r.standard_normal((T, H)) * 4e-3).astype(np.float32)
    hd, bd, rd = torch.from_numpy(h).to(device), U.to_device(branch, "bf16", device), torch.from_numpy(ref).to(device)
    out = torch.empty(T, H, dtype=torch.float32, device=device)
    d_out = torch.empty(T, H, dtype=torch.bfloat16, device=device)
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    ws = C.workspace(C.catq_recon_loss_workspace_bytes(T * H), device)
    C.catq_block_output_loss(hd, bd, rd, loss, d_out, out, ws, reduction=reduction)
    want_out = h.astype(np.float64) + branch
    assert U.max_rel(_f32(out), want_out) <= 1e-7
    want_loss, want_d = O.recon_loss(want_out, ref, reduction)
    assert abs(loss.item() - want_loss) <= 1e-4 * want_loss  # fp32 differences of 4e-3 at magnitude 4
    assert U.fro_rel(_f32(d_out), want_d) <= U.TOL_BF16
    # the teacher's call: out only
    out2 = torch.zeros_like(out)
    C.catq_block_output_loss(hd, bd, out=out2)
    torch.cuda.synchronize()
    assert torch.equal(out, out2)


# ---------------------------------------------------------------- attention

# d = 128 with S a multiple of 128 takes the tcgen05 forward; the others the mma.sync one
ATTN_SHAPES = [(2, 128, 4, 2, 128), (1, 192, 4, 1, 64), (1, 64, 2, 2, 128), (3, 256, 8, 8, 64), (2, 512, 8, 2, 128),
               (1, 384, 4, 4, 128)]


def _attn_inputs(B, S, nh, nkv, d, tag):
    r = syn.rng(95, tag)
    return (_bf16(r, (B * S, nh * d)), _bf16(r, (B * S, nkv * d)), _bf16(r, (B * S, nkv * d)),
            _bf16(r, (B * S, nh * d)))


def _gpu_attention(q, k, v, do, B, S, nh, nkv, d, device):
    import torch

    from paper_2606_26650_gb300 import catq as C
    qd, kd, vd, dod = (U.to_device(a, "bf16", device) for a in (q, k, v, do))
    o = torch.empty_like(qd)
    lse = torch.empty(B * nh * S, dtype=torch.float32, device=device)
    C.catq_attention_fwd(qd, kd, vd, o, lse, B, S, nh, nkv, d)
    dq, dk, dv = torch.empty_like(qd), torch.empty_like(kd), torch.empty_like(vd)
    delta = torch.empty_like(lse)
    C.catq_attention_bwd(qd, kd, vd, o, dod, lse, delta, dq, dk, dv, B, S, nh, nkv, d)
    torch.cuda.synchronize()
    return {n: _f32(t) for n, t in (("o", o), ("lse", lse), ("dq", dq), ("dk", dk), ("dv", dv))}


@pytest.mark.parametrize("B,S,nh,nkv,d", ATTN_SHAPES)
def test_attention_fwd_bwd(device, B, S, nh, nkv, d):
    q, k, v, do = _attn_inputs(B, S, nh, nkv, d, f"attn/{B}/{S}/{nh}/{nkv}/{d}")
    got = _gpu_attention(q, k, v, do, B, S, nh, nkv, d, device)
    o, p = O.attention(q, k, v, B, S, nh, nkv, d)
    lse = O.attention_logsumexp(q, k, B, S, nh, nkv, d)
    dq, dk, dv = O.attention_bwd(q, k, v, p, do, B, S, nh, nkv, d)
    assert np.abs(got["lse"] - lse.ravel()).max() <= 1e-4
    errs = {n: U.fro_rel(got[n], w) for n, w in (("o", o), ("dq", dq), ("dk", dk), ("dv", dv))}
    assert all(e <= U.TOL_BF16 for e in errs.values()), errs


def test_attention_full_size_sampled(device):
    """The Llama-3-8B block's attention at full size; the oracle computes every row of
    sequence 3's key/value head 5 (query heads 20..23)."""
    B, S, nh, nkv, d = 4, 2048, 32, 8, 128
    q, k, v, do = _attn_inputs(B, S, nh, nkv, d, "attn/full")
    got = _gpu_attention(q, k, v, do, B, S, nh, nkv, d, device)
    b, hk, rep = 3, 5, nh // nkv
    rows = slice(b * S, (b + 1) * S)
    qs = q[rows, hk * rep * d:(hk + 1) * rep * d]
    dos = do[rows, hk * rep * d:(hk + 1) * rep * d]
    ks, vs = k[rows, hk * d:(hk + 1) * d], v[rows, hk * d:(hk + 1) * d]
    o, p = O.attention(qs, ks, vs, 1, S, rep, 1, d)
    lse = O.attention_logsumexp(qs, ks, 1, S, rep, 1, d)
    dq, dk, dv = O.attention_bwd(qs, ks, vs, p, dos, 1, S, rep, 1, d)
    del p
    cols = slice(hk * rep * d, (hk + 1) * rep * d)
    lse_got = got["lse"].reshape(B, nh, S)[b, hk * rep:(hk + 1) * rep]
    assert np.abs(lse_got - lse[0]).max() <= 1e-4
    errs = {"o": U.fro_rel(got["o"][rows, cols], o), "dq": U.fro_rel(got["dq"][rows, cols], dq),
            "dk": U.fro_rel(got["dk"][rows, hk * d:(hk + 1) * d], dk),
            "dv": U.fro_rel(got["dv"][rows, hk * d:(hk + 1) * d], dv)}
    assert all(e <= U.TOL_BF16 for e in errs.values()), errs


# ---------------------------------------------------------------- the block step

SMALL = dict(H=512, n_heads=4, n_kv_heads=2, d=128, I=1024, B=2, S=128, base=500000.0, eps=1e-5)


def _block_case(shape, g, seed, x_dtype="bf16"):
    r = syn.rng(96, f"block/{seed}")
    W = {n: _bf16(r, (N, K), 0.02) for n, (N, K) in shape.linear_shapes().items()}
    x = (r.standard_t(4.0, (shape.T, shape.H))).astype(np.float32)
    if x_dtype == "bf16":
        x = syn.round_bf16(x)
    g1 = r.uniform(0.5, 1.5, shape.H).astype(np.float32)
    g2 = r.uniform(0.5, 1.5, shape.H).astype(np.float32)
    fac = {n: syn.factors(W[n].size // g, seed, f"block/{n}", perturbed=True) for n in W}
    return W, x, g1, g2, fac


def _gpu_block(shape, W, x, g1, g2, fac, g, phase, s, device, x_dtype="bf16", qk=None, side_streams=3):
    import torch

    from paper_2606_26650_gb300 import block as BK
    from paper_2606_26650_gb300 import catq as C
    Wd = {n: U.to_device(w, "bf16", device) for n, w in W.items()}
    facd = {n: tuple(torch.from_numpy(f.copy()).to(device) for f in fac[n]) for n in W}
    norms = {k: torch.from_numpy(v).to(device) for k, v in qk.items()} if qk else {}
    blk = BK.Block(shape, Wd, torch.from_numpy(g1).to(device), torch.from_numpy(g2).to(device), g, factors=facd,
                   side_streams=side_streams, **norms)
    xd = U.to_device(x, x_dtype, device)
    out_ref = torch.empty(shape.T, shape.H, dtype=torch.float32, device=device)
    blk.teacher(xd, out_ref)
    out = torch.empty_like(out_ref)
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    grads = {n: [torch.empty(W[n].size // g, dtype=torch.float32, device=device) for _ in range(3)] for n in W}
    blk.step(xd, out_ref, C.schedule(phase, s), loss, grads, out=out)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    return dict(out_ref=_f32(out_ref), out=_f32(out), loss=loss.item(),
                g={n: tuple(_f32(t) for t in grads[n]) for n in W})


@pytest.mark.parametrize("phase,s,x_dtype,qk_norm", [(O.PHASE_SOFT, 30.0, "bf16", False),
                                                     (O.PHASE_SOFT, 0.625, "bf16", False),
                                                     (O.PHASE_HARD, 30.0, "bf16", False),
                                                     (O.PHASE_SOFT, 30.0, "f32", False),
                                                     (O.PHASE_SOFT, 30.0, "bf16", True),
                                                     (O.PHASE_HARD, 30.0, "bf16", True)])
def test_block_step_matches_oracle(device, phase, s, x_dtype, qk_norm):
    """qk_norm: the Qwen3 block (per-head query/key RMSNorm, RoPE base 1e6)."""
    from paper_2606_26650_gb300 import block as BK
    shape = BK.BlockShape(**dict(SMALL, base=1e6 if qk_norm else SMALL["base"]))
    g = 128
    W, x, g1, g2, fac = _block_case(shape, g, 1, x_dtype)
    qk = None
    if qk_norm:
        rq = syn.rng(99, "block/qk")
        qk = {"q_norm": rq.uniform(0.5, 1.5, shape.d).astype(np.float32),
              "k_norm": rq.uniform(0.5, 1.5, shape.d).astype(np.float32)}
    got = _gpu_block(shape, W, x, g1, g2, fac, g, phase, s, device, x_dtype, qk=qk)
    stats = {n: O.group_stats(W[n], g) for n in W}
    ref = O.block_calibration_step(x, W, g, stats, fac, g1, g2, shape.B, shape.S, shape.n_heads, shape.n_kv_heads,
                                   shape.d, shape.base, shape.eps, phase, s, **(qk or {}))
    errs = {"out_ref": U.fro_rel(got["out_ref"], ref["out_ref"]), "out": U.fro_rel(got["out"], ref["out"]),
            "out-out_ref": U.fro_rel(got["out"] - got["out_ref"], ref["out"] - ref["out_ref"]),
            "loss": abs(got["loss"] - ref["loss"]) / ref["loss"]}
    for n in W:
        for name, a, b in zip(("g_dmu", "g_dalpha", "g_ddelta"), got["g"][n], ref["g"][n]):
            errs[f"{n}.{name}"] = U.fro_rel(a, b)
    print("block step errors:", {k: f"{v:.2e}" for k, v in errs.items()})
    bad = {k: v for k, v in errs.items() if not v <= U.TOL_BF16}
    assert not bad, f"tolerance {U.TOL_BF16} exceeded: {bad}"


@pytest.mark.parametrize("qk_norm", [False, True])
def test_block_step_same_on_any_number_of_streams(device, qk_norm):
    """Every kernel of the step is deterministic, and the side streams only change which calls
    overlap: the step on the main stream alone, on one side stream and on three gives the same
    bits (the events order every read after its write)."""
    from paper_2606_26650_gb300 import block as BK
    shape = BK.BlockShape(**dict(SMALL, base=1e6 if qk_norm else SMALL["base"]))
    W, x, g1, g2, fac = _block_case(shape, 128, 3)
    qk = None
    if qk_norm:
        rq = syn.rng(99, "block/qk")
        qk = {"q_norm": rq.uniform(0.5, 1.5, shape.d).astype(np.float32),
              "k_norm": rq.uniform(0.5, 1.5, shape.d).astype(np.float32)}
    runs = [_gpu_block(shape, W, x, g1, g2, fac, 128, O.PHASE_SOFT, 30.0, device, qk=qk, side_streams=n)
            for n in (0, 1, 3)]
    for r in runs[1:]:
        assert np.array_equal(r["out"], runs[0]["out"])
        assert r["loss"] == runs[0]["loss"]
        for n in W:
            for a, b in zip(r["g"][n], runs[0]["g"][n]):
                assert np.array_equal(a, b), n


def test_block_teacher_phase_has_zero_loss(device):
    """At the TEACHER phase the student is the teacher: the same kernels on the same inputs
    give the same output, so the loss is exactly 0 and every factor gradient 0."""
    from paper_2606_26650_gb300 import block as BK
    shape = BK.BlockShape(**dict(SMALL, S=64, B=1))
    W, x, g1, g2, fac = _block_case(shape, 128, 2)
    got = _gpu_block(shape, W, x, g1, g2, fac, 128, O.PHASE_TEACHER, 0.0, device)
    assert got["loss"] == 0.0
    assert np.array_equal(got["out"], got["out_ref"])
    assert all(np.all(t == 0.0) for n in got["g"] for t in got["g"][n])


def test_block_calibration_loop_matches_oracle(device):
    """The block window's calibration loop (§8(f) row 1): epochs of block steps under the
    epoch schedule of Eq. 6 (SOFT epochs of rising sharpness, then HARD), each followed by
    AdamW on every linear's three factors at the linearly decayed learning rate, on the GPU
    and in the oracle from the same seeded block.  Per-step losses within 2e-2 and each
    linear's factor movement (end minus start) within 2e-2 relative Frobenius error, the bar of
    the gradients the loop integrates; the loss falls on both sides."""
    import torch

    from paper_2606_26650_gb300 import block as BK
    from paper_2606_26650_gb300 import catq as C
    shape = BK.BlockShape(**dict(SMALL, S=64))
    g, batches, m, gamma, s0, lr0 = 128, 2, 6, 4 / 6, 30.0, 1e-3
    W, _, g1, g2, _ = _block_case(shape, g, 3)
    r = syn.rng(98, "block_loop")
    xs = [syn.round_bf16(r.standard_t(4.0, (shape.T, shape.H)).astype(np.float32)) for _ in range(batches)]
    G = {n: W[n].size // g for n in W}
    names = list(BK.LINEARS)
    # oracle loop
    stats = {n: O.group_stats(W[n], g) for n in names}
    fac = {n: (np.zeros(G[n]), np.ones(G[n]), np.ones(G[n])) for n in names}
    mom = {n: (np.zeros(G[n]),) * 6 for n in names}
    losses_o, t = [], 0
    for e in range(1, m + 1):
        phase, s = O.schedule_at_epoch(e, m, gamma, s0)
        for x in xs:
            step = O.block_calibration_step(x, W, g, stats, fac, g1, g2, shape.B, shape.S, shape.n_heads,
                                            shape.n_kv_heads, shape.d, shape.base, shape.eps, phase, s)
            losses_o.append(step["loss"])
            lr = O.linear_decay_lr(lr0, t, m * batches)
            t += 1
            for n in names:
                fac[n], mom[n] = O.factor_update(fac[n], step["g"][n], mom[n], t, lr)
    # GPU loop
    Wd = {n: U.to_device(w, "bf16", device) for n, w in W.items()}
    blk = BK.Block(shape, Wd, torch.from_numpy(g1).to(device), torch.from_numpy(g2).to(device), g)
    xds = [U.to_device(x, "bf16", device) for x in xs]
    refs = []
    for xd in xds:
        o = torch.empty(shape.T, shape.H, dtype=torch.float32, device=device)
        blk.teacher(xd, o)
        refs.append(o)
    grads = {n: [torch.empty(G[n], dtype=torch.float32, device=device) for _ in range(3)] for n in names}
    moments = {n: torch.zeros(6 * G[n], dtype=torch.float32, device=device) for n in names}
    hp = C.adamw()
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    losses_g = torch.zeros(m * batches, dtype=torch.float32, device=device)
    t = 0
    for e in range(1, m + 1):
        sched = C.catq_schedule_at_epoch(e, m, gamma, s0)
        for xd, ref in zip(xds, refs):
            blk.step(xd, ref, sched, loss, grads)
            losses_g[t].copy_(loss[0])
            lr = C.catq_linear_decay_lr(lr0, t, m * batches)
            t += 1
            for n in names:
                L = blk.layers[n]
                C.catq_factor_adamw_step(L.d_mu, L.d_alpha, L.d_delta, *grads[n], moments[n], hp, t, lr)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    lg, lo = U.to_host(losses_g).astype(np.float64), np.array(losses_o)
    rel = np.abs(lg - lo) / np.abs(lo)
    moves = {}
    for n in names:
        L = blk.layers[n]
        start = (np.zeros(G[n]), np.ones(G[n]), np.ones(G[n]))
        got = tuple(U.to_host(f).astype(np.float64) for f in (L.d_mu, L.d_alpha, L.d_delta))
        for name, a, b, s0_ in zip(("d_mu", "d_alpha", "d_delta"), got, fac[n], start):
            moves[f"{n}.{name}"] = U.fro_rel(a - s0_, b - s0_)
    print(f"block loop: worst step loss error {rel.max():.3e}, worst factor movement error "
          f"{max(moves.values()):.3e}, loss {lo[0]:.4e} -> {lo[-1]:.4e}")
    assert rel.max() <= U.TOL_BF16, rel
    bad = {k: v for k, v in moves.items() if not v <= U.TOL_BF16}
    assert not bad, bad
    assert lo[-1] < lo[0] and lg[-1] < lg[0]


def test_block_full_size_sampled(device):
    """The Llama-3-8B block window at full size (4 x 2048 tokens), in the launch configuration
    the bench times.  At the TEACHER phase the loss is exactly 0 and every factor gradient 0.
    In the SOFT phase (s = 30) the factor gradients of q_proj and down_proj (the first and last
    linears of the backward) are checked on 2 sampled W rows of every 256-row block, against
    the oracle's chain rule (Eq. 3, 5, 6) applied to G = dY^T X formed in fp64 from the GPU's
    own dY and X of that linear inside the block (so the check isolates the block's dW path at
    full size; the layers upstream are checked at reduced size above).  Within 1e-3 relative
    Frobenius error per linear and factor."""
    import torch

    from paper_2606_26650_gb300 import block as BK
    from paper_2606_26650_gb300 import catq as C
    wl = syn.WORKLOADS["c3_llama3_8b_block"]
    shape = BK.BlockShape(H=4096, n_heads=32, n_kv_heads=8, d=128, I=14336, B=4, S=2048)
    g = wl.g
    Wh = {lin.name: syn.weight(wl, lin) for lin in wl.linears}
    W = {n: U.to_device(w, "bf16", device) for n, w in Wh.items()}
    fac = {n: syn.factors(Wh[n].size // g, 0, f"block_full/{n}", perturbed=True) for n in Wh}
    r = syn.rng(100, "block_full")
    g1, g2 = (r.uniform(0.5, 1.5, shape.H).astype(np.float32) for _ in range(2))
    blk = BK.Block(shape, W, torch.from_numpy(g1).to(device), torch.from_numpy(g2).to(device), g,
                   factors={n: tuple(torch.from_numpy(f.copy()).to(device) for f in fac[n]) for n in Wh})
    x = U.to_device(syn.activations(wl, "x_hidden", shape.T, shape.H), "bf16", device)
    out_ref = torch.empty(shape.T, shape.H, dtype=torch.float32, device=device)
    blk.teacher(x, out_ref)
    loss = torch.zeros(1, dtype=torch.float32, device=device)
    grads = {n: [torch.empty(Wh[n].size // g, dtype=torch.float32, device=device) for _ in range(3)] for n in Wh}
    blk.step(x, out_ref, C.schedule(C.PHASE_TEACHER), loss, grads)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    assert loss.item() == 0.0
    assert all(int(torch.count_nonzero(t).item()) == 0 for n in grads for t in grads[n])
    s = 30.0
    blk.step(x, out_ref, C.schedule(C.PHASE_SOFT, s), loss, grads)
    torch.cuda.synchronize()
    assert C.catq_device_status() == 0
    assert np.isfinite(loss.item()) and loss.item() > 0.0
    rs = syn.rng(101, "block_full/rows")
    for name, X_t, dY_t in (("q_proj", blk.z1, blk.dq), ("down_proj", blk.m, blk.d_out)):
        Wn = Wh[name]
        N, K = Wn.shape
        rows = np.sort(np.concatenate([rs.choice(np.arange(b, min(b + 256, N)), 2, replace=False)
                                       for b in range(0, N, 256)]))
        Xh = U.to_host(X_t).astype(np.float64)
        dYh = U.to_host(dY_t).astype(np.float64)[:, rows]
        Gw = dYh.T @ Xh                           # [rows, K], fp64
        gpr = K // g
        gidx = (rows[:, None] * gpr + np.arange(gpr)[None, :]).ravel()
        stats = O.group_stats(Wn[rows], g)
        f_rows = tuple(f[gidx] for f in fac[name])
        want = O.factor_grads_from_G(Gw, Wn[rows], g, stats, f_rows, O.PHASE_SOFT, s)
        got = [U.to_host(t).astype(np.float64)[gidx] for t in grads[name]]
        errs = {q: U.fro_rel(a, b) for q, a, b in zip(("g_dmu", "g_dalpha", "g_ddelta"), got, want)}
        print(name, {k: f"{v:.2e}" for k, v in errs.items()})
        assert all(v <= 1e-3 for v in errs.values()), (name, errs)
