"""The C-ABI library without a GPU: it loads, exports every function include/catq.h
declares, and rejects bad arguments on the host before anything reaches a device."""
import ctypes
import os

import pytest

from paper_2606_26650_gb300 import catq as C


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(C.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    return C.lib()


def test_exports_every_declared_symbol(lib):
    names = C.header_functions()
    assert len(names) >= 11
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings_and_version(lib):
    assert lib.catq_abi_version() == 3
    for code, name in C.STATUS.items():
        assert lib.catq_status_string(code).decode() == name
    assert lib.catq_status_string(99).decode() == "CATQ_ERR_UNKNOWN"


def _layer(N=64, K=256, g=128, dtype=C.BF16, W=16, stats=32, op_const=65536, recon=C.RECON_ALPHA_T, reserved=0):
    """A layer struct with fake (never dereferenced) device addresses."""
    return C.catq_layer(N, K, g, dtype, W, stats, stats + 1024, stats + 2048, stats + 4096, stats + 8192,
                        stats + 16384, op_const, recon, reserved)


def _stats(lib, layer, thr=0):
    return lib.catq_group_stats(ctypes.byref(layer), thr, None)


def test_layer_validation(lib):
    assert lib.catq_group_stats(None, 0, None) == 1
    assert _stats(lib, _layer(W=0)) == 1                     # null W
    assert _stats(lib, _layer(K=250)) == 2                   # g does not divide K
    assert _stats(lib, _layer(g=32)) == 2                    # bf16 needs g % 64 == 0
    assert _stats(lib, _layer(N=60)) == 2                    # bf16 needs N % 8 == 0
    assert _stats(lib, _layer(g=48, K=96, dtype=C.F32)) == 2  # fp32 g not supported
    assert _stats(lib, _layer(dtype=7)) == 3                 # unknown dtype
    assert _stats(lib, _layer(W=24)) == 4                    # misaligned W
    assert _stats(lib, _layer(), thr=5) == 1                 # bad threshold rule
    assert _stats(lib, _layer(N=0)) == 2
    assert _stats(lib, _layer(recon=2)) == 1                 # unknown reconstruction
    assert _stats(lib, _layer(reserved=1)) == 1              # reserved field must be 0


def test_call_validation(lib):
    L = _layer()
    soft = C.schedule(C.PHASE_SOFT, 30.0)
    fwd = lib.catq_soft_ternary_linear_fwd
    assert fwd(ctypes.byref(L), C.schedule(9, 1.0), 16, 4, C.BF16, 16, None) == 1      # bad phase
    assert fwd(ctypes.byref(L), C.schedule(C.PHASE_SOFT, 0.0), 16, 4, C.BF16, 16, None) == 1  # s must be > 0
    assert fwd(ctypes.byref(L), C.schedule(C.PHASE_SOFT, float("nan")), 16, 4, C.BF16, 16, None) == 1
    assert fwd(ctypes.byref(L), soft, 16, 4, C.F32, 16, None) == 3                   # mixed dtypes
    assert fwd(ctypes.byref(L), soft, 16, -1, C.BF16, 16, None) == 2                 # M < 0
    assert fwd(ctypes.byref(L), soft, 16, 0, C.BF16, 16, None) == 0                  # M == 0: no-op
    assert fwd(ctypes.byref(L), soft, 0, 4, C.BF16, 16, None) == 1                   # null X
    assert fwd(ctypes.byref(L), soft, 24, 4, C.BF16, 16, None) == 4                  # misaligned X
    # a bf16 SOFT/HARD forward or dX needs the operand-constant array, 16-byte aligned
    assert fwd(ctypes.byref(_layer(op_const=0)), soft, 16, 4, C.BF16, 16, None) == 1
    assert fwd(ctypes.byref(_layer(op_const=65544)), soft, 16, 4, C.BF16, 16, None) == 4
    assert lib.catq_soft_ternary_linear_bwd(ctypes.byref(_layer(op_const=0)), soft, 16, 16, 4, C.BF16, 16,
                                            None, None, None, None, 0, None) == 1
    bwd = lib.catq_soft_ternary_linear_bwd
    assert bwd(ctypes.byref(L), soft, 16, 16, 4, C.BF16, None, 0, 32, 32, 256, 1 << 30, None) == 1
    F = _layer(dtype=C.F32)
    need = lib.catq_bwd_workspace_bytes(ctypes.byref(F), 4)
    assert need == 3 * 64 * (256 // 64) * 4
    assert bwd(ctypes.byref(F), soft, 16, 16, 4, C.F32, None, 32, 32, 32, 256, need - 1, None) == 9
    assert bwd(ctypes.byref(F), soft, 16, 16, 4, C.F32, None, 32, 32, 32, 0, need, None) == 9
    assert bwd(ctypes.byref(F), soft, 16, 16, 4, C.F32, None, 32, 32, 32, 128, need, None) == 4
    loss = lib.catq_recon_loss
    ws = lib.catq_recon_loss_workspace_bytes(1000)
    assert ws >= 8 and ws % 256 == 0
    assert loss(16, 16, 1000, 5, 0, 16, None, 256, ws, None) == 3
    assert loss(16, 16, 1000, C.BF16, 2, 16, None, 256, ws, None) == 1
    assert loss(16, 16, 0, C.BF16, 0, 16, None, 256, ws, None) == 2
    assert loss(16, 16, 1000, C.BF16, 0, 16, None, 256, ws - 256, None) == 9
    assert loss(16, 24, 1000, C.BF16, 0, 16, None, 256, ws, None) == 4
    pack = lib.catq_hard_ternarize_pack
    assert pack(ctypes.byref(L), None, None, None, None) == 1
    assert lib.catq_device_status(None, None) == 1
    infer = lib.catq_ternary_infer
    assert infer(None, 32, None, 64, 256, 128, 16, 1, C.BF16, 16, None) == 1       # null codes
    assert infer(16, 32, None, 64, 256, 128, 16, 1, C.F32, 16, None) == 3           # bf16 only
    assert infer(16, 32, None, 64, 256, 32, 16, 1, C.BF16, 16, None) == 2           # g % 64 != 0
    assert infer(16, 32, None, 64, 250, 128, 16, 1, C.BF16, 16, None) == 2          # g does not divide K
    assert infer(16, 32, None, 64, 256, 128, 16, 0, C.BF16, 16, None) == 0          # B == 0: no-op
    assert infer(24, 32, None, 64, 256, 128, 16, 1, C.BF16, 16, None) == 4          # misaligned codes
    assert infer(16, 32, 34, 64, 256, 128, 16, 1, C.BF16, 16, None) == 4            # misaligned mu
    assert infer(16, 32, None, 64, 256, 128, 16, 1, C.BF16, None, None) == 1        # null Y
    assert lib.catq_selftest_wait_timeout(10, None) == 1              # below 1 us
    assert lib.catq_selftest_wait_timeout(2_000_000_000, None) == 1   # above 1 s


def test_schedule_and_lr_host_calls_follow_the_oracle(lib):
    """The host-only schedule calls against the oracle: the branch exactly, s and the
    learning rate to fp32 rounding."""
    from oracle import catq_oracle as O
    for m, gamma, s0 in [(60, 0.8, 30.0), (10, 1.0, 5.0), (7, 0.5, 12.0), (100, 0.57, 30.0), (1, 0.3, 2.0),
                          (10, 0.75, 30.0), (3, 0.2, 30.0)]:
        for e in range(m + 1):
            got = C.catq_schedule_at_epoch(e, m, gamma, s0)
            phase, s = O.schedule_at_epoch(e, m, gamma, s0)
            assert got.phase == phase, (m, gamma, e)
            assert got.s == pytest.approx(s, rel=1e-7, abs=0.0), (m, gamma, e)
    for total in (1, 8, 10260):
        for k in sorted({0, 1, total // 2, total - 1}):
            if k < total:
                assert C.catq_linear_decay_lr(1e-3, k, total) == pytest.approx(O.linear_decay_lr(1e-3, k, total),
                                                                                rel=1e-7)


def test_schedule_and_update_validation(lib):
    out = C.catq_schedule()
    sched = lib.catq_schedule_at_epoch
    assert sched(1, 60, 0.8, 30.0, ctypes.byref(out)) == 0
    assert sched(61, 60, 0.8, 30.0, ctypes.byref(out)) == 1   # e > m
    assert sched(-1, 60, 0.8, 30.0, ctypes.byref(out)) == 1
    assert sched(0, 0, 0.8, 30.0, ctypes.byref(out)) == 1     # m < 1
    assert sched(1, 60, 0.0, 30.0, ctypes.byref(out)) == 1    # gamma outside (0, 1]
    assert sched(1, 60, 1.5, 30.0, ctypes.byref(out)) == 1
    assert sched(1, 60, 0.8, 0.0, ctypes.byref(out)) == 1     # s0 <= 0
    assert sched(1, 60, 0.8, float("inf"), ctypes.byref(out)) == 1
    assert sched(1, 60, 0.8, 30.0, None) == 1
    lr = ctypes.c_float()
    assert lib.catq_linear_decay_lr(1e-3, 5, 5, ctypes.byref(lr)) == 1  # k >= total
    assert lib.catq_linear_decay_lr(-1.0, 0, 5, ctypes.byref(lr)) == 1
    assert lib.catq_linear_decay_lr(float("nan"), 0, 5, ctypes.byref(lr)) == 1
    # the update rejects bad arguments on the host (fake, never dereferenced addresses)
    hp = C.adamw()
    step = lib.catq_factor_adamw_step
    ptrs = [4096 * (i + 1) for i in range(7)]
    assert step(-1, *ptrs, ctypes.byref(hp), 1, 1e-3, None) == 2
    assert step(0, *ptrs, ctypes.byref(hp), 1, 1e-3, None) == 0  # no work, nothing launched
    assert step(0, *([None] * 7), None, 0, -1.0, None) == 0
    assert step(8, *ptrs[:6], None, ctypes.byref(hp), 1, 1e-3, None) == 1
    assert step(8, *ptrs, None, 1, 1e-3, None) == 1
    assert step(8, *ptrs, ctypes.byref(hp), 0, 1e-3, None) == 1  # t < 1
    assert step(8, *ptrs, ctypes.byref(hp), 1, -1e-3, None) == 1
    assert step(8, *ptrs, ctypes.byref(hp), 1, float("nan"), None) == 1
    for bad in (C.adamw(beta1=1.0), C.adamw(beta2=-0.1), C.adamw(eps=0.0), C.adamw(weight_decay=-1.0),
                C.adamw(margin=0.5), C.adamw(eps=float("inf"))):
        assert step(8, *ptrs, ctypes.byref(bad), 1, 1e-3, None) == 1
    assert step(8, *ptrs[:6], ptrs[6] + 2, ctypes.byref(hp), 1, 1e-3, None) == 4  # misaligned moments


def test_block_call_validation(lib):
    """The decoder-block calls reject bad shapes, dtypes, scalars, null and misaligned
    pointers and short workspaces on the host, and treat empty inputs as no-ops, before any
    launch (fake device addresses, never dereferenced)."""
    inf, nan = float("inf"), float("nan")
    att = lib.catq_attention_fwd
    assert att(16, 16, 16, 1, 100, 8, 2, 128, 16, 16, None) == 2    # S % 64 != 0
    assert att(16, 16, 16, 1, 32, 8, 2, 128, 16, 16, None) == 2     # S < 64
    assert att(16, 16, 16, 1, 128, 8, 2, 96, 16, 16, None) == 2     # d not 64 or 128
    assert att(16, 16, 16, 1, 128, 6, 4, 128, 16, 16, None) == 2    # heads do not share evenly
    assert att(16, 16, 16, -1, 128, 8, 2, 128, 16, 16, None) == 2
    assert att(16, 16, 16, 70000, 128, 8, 2, 128, 16, 16, None) == 2
    assert att(None, None, None, 0, 128, 8, 2, 128, None, None, None) == 0  # B == 0: no-op
    assert att(None, 16, 16, 1, 128, 8, 2, 128, 16, 16, None) == 1  # null Q
    assert att(16, 16, 16, 1, 128, 8, 2, 128, 16, None, None) == 1  # null lse
    assert att(24, 16, 16, 1, 128, 8, 2, 128, 16, 16, None) == 4    # misaligned Q
    assert att(16, 16, 16, 1, 128, 8, 2, 128, 16, 18, None) == 4    # misaligned lse
    bwd = lib.catq_attention_bwd
    args = [16, 16, 16, 16, 16, 16, 1, 128, 8, 2, 128, 16, 16, 16, 16, None]
    assert bwd(*args[:10], 96, *args[11:]) == 2
    assert bwd(*args[:6], 0, *args[7:]) == 0                         # B == 0: no-op
    assert bwd(*args[:11], None, *args[12:]) == 1                    # null delta
    assert bwd(*args[:14], 40, None) == 4                            # misaligned dV
    assert bwd(*args[:11], 18, *args[12:]) == 4                      # misaligned delta

    rf = lib.catq_rmsnorm_fwd
    assert rf(16, 7, None, 16, 4, 64, 1e-5, None, 16, 16, None) == 3      # unknown dtype
    assert rf(16, C.BF16, None, 16, 4, 12, 1e-5, None, 16, 16, None) == 2  # H % 8 != 0
    assert rf(16, C.BF16, None, 16, -1, 64, 1e-5, None, 16, 16, None) == 2
    assert rf(16, C.BF16, None, 16, 4, 64, -1.0, None, 16, 16, None) == 1  # eps < 0
    assert rf(16, C.BF16, None, 16, 4, 64, nan, None, 16, 16, None) == 1
    assert rf(None, C.BF16, None, None, 0, 64, 1e-5, None, None, None, None) == 0  # T == 0
    assert rf(16, C.BF16, None, 16, 4, 64, 1e-5, None, None, 16, None) == 1  # null Z
    assert rf(16, C.BF16, 24, 16, 4, 64, 1e-5, None, 16, 16, None) == 4     # misaligned residual
    assert rf(16, C.BF16, None, 18, 4, 64, 1e-5, None, 16, 16, None) == 4   # misaligned gamma
    rb = lib.catq_rmsnorm_bwd
    assert rb(16, 5, 16, 16, 16, None, None, 4, 64, 16, None) == 3
    assert rb(16, C.F32, 16, 16, 16, None, None, 4, 0, 16, None) == 2      # H < 1
    assert rb(None, C.F32, None, None, None, None, None, 0, 64, None, None) == 0
    assert rb(16, C.F32, 16, 16, 16, None, None, 4, 64, None, None) == 1   # null dX
    assert rb(16, C.F32, 16, 16, 16, 24, None, 4, 64, 16, None) == 4       # misaligned dZ2

    rope = lib.catq_rope
    assert rope(16, 4, 4, 2, 7, 1e4, 0, None) == 2         # odd d
    assert rope(16, 4, 0, 2, 128, 1e4, 0, None) == 2       # S < 1
    assert rope(16, 4, 4, 2, 128, 1.0, 0, None) == 1       # base must exceed 1
    assert rope(16, 4, 4, 2, 128, inf, 0, None) == 1
    assert rope(None, 0, 4, 2, 128, 1e4, 0, None) == 0     # T == 0
    assert rope(None, 4, 4, 2, 128, 1e4, 0, None) == 1
    assert rope(24, 4, 4, 2, 128, 1e4, 0, None) == 4

    sf, sb = lib.catq_swiglu_fwd, lib.catq_swiglu_bwd
    assert sf(16, 16, -1, 16, None) == 2
    assert sf(None, None, 0, None, None) == 0
    assert sf(16, 16, 64, None, None) == 1
    assert sf(16, 24, 64, 16, None) == 4
    assert sb(16, 16, 16, 64, 16, None, None) == 1          # null d_up
    assert sb(16, 16, 24, 64, 16, 16, None) == 4            # misaligned dM

    bl = lib.catq_block_output_loss
    need = lib.catq_recon_loss_workspace_bytes(64)
    assert bl(16, 16, 12, 16, 0, 16, None, None, 256, need, None) == 2      # count % 8 != 0
    assert bl(16, 16, 64, 16, 3, 16, None, None, 256, need, None) == 1      # unknown reduction
    assert bl(None, None, 0, None, 0, None, None, None, None, 0, None) == 0  # count == 0
    assert bl(16, 16, 64, 16, 0, None, None, None, 256, need, None) == 1    # out_ref without loss_out
    assert bl(16, 24, 64, 16, 0, 16, None, None, 256, need, None) == 4      # misaligned branch
    assert bl(16, 16, 64, 16, 0, 16, None, None, 256, need - 8, None) == 9  # short workspace
    assert bl(16, 16, 64, 16, 0, 16, None, None, None, need, None) == 9     # no workspace
    assert bl(16, 16, 64, 16, 0, 16, None, None, 128, need, None) == 4      # workspace not 256-aligned


def _grouped(E=4, N=64, K=256, g=128, dtype=C.BF16, W=16, stats=32, op_const=65536, recon=C.RECON_ALPHA_T):
    """A stacked (MoE) layer struct with fake (never dereferenced) device addresses."""
    return C.catq_grouped_layer(E, g, N, K, dtype, recon, W, stats, stats + 1024, stats + 2048, stats + 4096,
                                stats + 8192, stats + 16384, op_const)


def _offsets(*rows):
    return (ctypes.c_int64 * len(rows))(*rows)


def test_linear_variant_call_validation(lib):
    """fwd_ex, fwd_loss, modulate_ternarize, act_quant_a8, the allocation-free backward and the
    per-group reconstruction error: host-side rejections and no-ops (fake device addresses)."""
    L, soft = _layer(), C.schedule(C.PHASE_SOFT, 30.0)
    ex = lib.catq_soft_ternary_linear_fwd_ex
    assert ex(ctypes.byref(L), soft, 16, 4, C.BF16, None, 16, 7, None) == 3     # Y dtype neither X's nor fp32
    assert ex(ctypes.byref(L), soft, 16, 0, C.BF16, None, 16, C.F32, None) == 0  # M == 0
    assert ex(ctypes.byref(L), soft, 16, 4, C.BF16, 18, 16, C.F32, None) == 4    # misaligned row scales
    assert ex(ctypes.byref(L), soft, 16, 4, C.BF16, None, None, C.F32, None) == 1
    fl = lib.catq_soft_ternary_linear_fwd_loss
    ok = [ctypes.byref(L), soft, 16, 4, C.BF16, None, 16, C.BF16, 0, 16, 16, None, 256, 1 << 20, None]
    assert fl(*ok[:7], 5, *ok[8:]) == 3                       # reference dtype
    assert fl(*ok[:8], 2, *ok[9:]) == 1                       # unknown reduction
    assert fl(*ok[:3], 0, *ok[4:]) == 2                       # M < 1
    assert fl(*ok[:10], None, *ok[11:]) == 1                  # null dY
    assert fl(*ok[:11], 24, *ok[12:]) == 4                    # misaligned Y
    assert fl(*ok[:12], None, *ok[13:]) == 9                  # no workspace
    mt = lib.catq_modulate_ternarize
    assert mt(ctypes.byref(_layer(stats=32)), C.schedule(C.PHASE_SOFT, -1.0), 16, None, None, None) == 1
    assert mt(ctypes.byref(L), soft, 24, None, None, None) == 4                 # misaligned Wq
    assert mt(ctypes.byref(L), soft, None, 40, None, None) == 4                 # misaligned codes
    assert mt(ctypes.byref(L), soft, None, None, None, None) == 0               # nothing asked for
    aq = lib.catq_act_quant_a8
    assert aq(16, 4, 256, 5, 16, 16, None, None) == 3
    assert aq(16, 4, 0, C.BF16, 16, 16, None, None) == 2      # K < 1
    assert aq(16, 4, 12, C.BF16, 16, 16, None, None) == 2     # bf16 rows of 16 bytes
    assert aq(16, 4, 6, C.F32, 16, 16, None, None) == 2       # fp32 rows of 16 bytes
    assert aq(None, 0, 256, C.BF16, None, None, None, None) == 0
    assert aq(16, 4, 256, C.BF16, 16, None, None, None) == 1  # null scales
    assert aq(16, 4, 256, C.BF16, 16, 18, None, None) == 4    # misaligned scales
    assert aq(16, 4, 256, C.BF16, 16, 16, 24, None) == 4      # misaligned dequantized copy
    na = lib.catq_soft_ternary_linear_bwd_noalloc
    assert lib.catq_bwd_noalloc_max_scratch_bytes() == 16 << 20
    assert na(ctypes.byref(_layer(W=0)), soft, 16, 16, 4, C.BF16, None, 32, 32, 32, None) == 1
    big = _layer(N=16384, K=16384, dtype=C.F32)                # 50 MB of partial sums
    assert na(ctypes.byref(big), soft, 16, 16, 4, C.F32, None, 32, 32, 32, None) == 9
    re = lib.catq_group_recon_error
    assert re(ctypes.byref(L), None, None) == 1
    assert re(ctypes.byref(L), 18, None) == 4
    assert re(ctypes.byref(_layer(dtype=9)), 16, None) == 3


def test_grouped_call_validation(lib):
    """The stacked-expert calls: offsets start at 0 and never decrease, dtype and workspace
    rules, empty routing as a no-op, and the grouped partial-sum size."""
    G, soft = _grouped(), C.schedule(C.PHASE_SOFT, 30.0)
    off = _offsets(0, 5, 5, 40, 64)
    fwd = lib.catq_grouped_soft_ternary_linear_fwd
    assert fwd(None, soft, 16, off, C.BF16, 16, None) == 1
    assert fwd(ctypes.byref(_grouped(E=0)), soft, 16, off, C.BF16, 16, None) == 1
    assert fwd(ctypes.byref(G), soft, 16, _offsets(1, 5, 5, 40, 64), C.BF16, 16, None) == 2  # off[0] != 0
    assert fwd(ctypes.byref(G), soft, 16, _offsets(0, 5, 4, 40, 64), C.BF16, 16, None) == 2  # decreasing
    assert fwd(ctypes.byref(G), soft, 16, _offsets(0, 0, 0, 0, 0), C.BF16, 16, None) == 0    # nothing routed
    assert fwd(ctypes.byref(G), soft, None, off, C.BF16, 16, None) == 1
    assert fwd(ctypes.byref(G), soft, 24, off, C.BF16, 16, None) == 4
    assert fwd(ctypes.byref(_grouped(op_const=0)), soft, 16, off, C.BF16, 16, None) == 1  # operand constants
    fl = lib.catq_grouped_soft_ternary_linear_fwd_loss
    ok = [ctypes.byref(G), soft, 16, off, C.BF16, 16, 0, 16, 16, None, 256, 1 << 20, None]
    assert fl(*ok[:4], C.F32, *ok[5:]) == 3
    assert fl(*ok[:6], 2, *ok[7:]) == 1
    assert fl(ok[0], soft, 16, _offsets(0, 0, 0, 0, 0), *ok[4:]) == 2   # loss over no rows
    assert fl(*ok[:8], None, *ok[9:]) == 1                               # null dY
    assert fl(*ok[:9], 24, *ok[10:]) == 4                                # misaligned Y
    assert fl(*ok[:10], None, *ok[11:]) == 9
    assert lib.catq_grouped_fwd_loss_workspace_bytes(ctypes.byref(G), _offsets(2, 5, 5, 40, 64)) == 0
    need = lib.catq_grouped_bwd_workspace_bytes(ctypes.byref(G), off)
    assert need == 4 * 3 * 64 * (256 // 128) * 4                         # [E][3][N][K/128] fp32
    assert lib.catq_grouped_bwd_workspace_bytes(None, off) == 0
    bwd = lib.catq_grouped_soft_ternary_linear_bwd
    ok = [ctypes.byref(G), soft, 16, 16, off, C.BF16, None, 32, 32, 32, 256, need, None]
    assert bwd(*ok[:8], None, *ok[9:]) == 1                              # all three gradients or none
    assert bwd(*ok[:2], None, *ok[3:]) == 1                              # null X
    assert bwd(*ok[:3], 24, *ok[4:]) == 4                                # misaligned dY
    assert bwd(*ok[:10], None, *ok[11:]) == 9
    assert bwd(*ok[:11], need - 4, None) == 9
    assert bwd(*ok[:10], 128, *ok[11:]) == 4                             # workspace not 256-aligned


def test_batched_and_staged_inference_validation(lib):
    """Layer lists of the batched and staged decode calls: limits, shared g and mu presence,
    the stage map, and the synchronisation words."""
    n_max, s_max = lib.catq_ternary_infer_max_layers(), lib.catq_ternary_infer_max_stages()
    assert 1 <= n_max <= 64 and s_max >= 1
    assert lib.catq_ternary_infer_sync_bytes() == 4 * (s_max + 1)

    def layers(n=2, mu=None, K=256, X=16, codes=16):
        arr = (C.catq_infer_layer * n)()
        for i in range(n):
            arr[i] = C.catq_infer_layer(codes, 32, mu, 64, K, X, 64)
        return arr
    bt = lib.catq_ternary_infer_batched
    assert bt(None, 2, 128, 1, C.BF16, None) == 1
    assert bt(layers(), 0, 128, 1, C.BF16, None) == 1
    assert bt(layers(n_max + 1), n_max + 1, 128, 1, C.BF16, None) == 1   # more layers than one launch takes
    assert bt(layers(), 2, 128, 1, C.F32, None) == 3
    assert bt(layers(), 2, 96, 1, C.BF16, None) == 2                     # g % 64 != 0
    assert bt(layers(K=320), 2, 128, 1, C.BF16, None) == 2               # g does not divide K
    mixed = layers()
    mixed[1].mu = 64
    assert bt(mixed, 2, 128, 1, C.BF16, None) == 1                       # mu on some layers only
    assert bt(layers(X=None), 2, 128, 1, C.BF16, None) == 1
    assert bt(layers(X=None), 2, 128, 0, C.BF16, None) == 0              # B == 0: inputs not needed
    assert bt(layers(codes=24), 2, 128, 1, C.BF16, None) == 4
    st = lib.catq_ternary_infer_staged
    stages = lambda *s: (ctypes.c_int32 * len(s))(*s)
    assert st(layers(3), 3, None, 128, 1, C.BF16, 64, None) == 1
    assert st(layers(3), 3, stages(0, 0, 1), 128, 1, C.BF16, None, None) == 1   # no sync words
    assert st(layers(3), 3, stages(1, 1, 2), 128, 1, C.BF16, 64, None) == 1    # first stage not 0
    assert st(layers(3), 3, stages(0, 2, 2), 128, 1, C.BF16, 64, None) == 1    # a stage skipped
    assert st(layers(3), 3, stages(0, 1, 0), 128, 1, C.BF16, 64, None) == 1    # stages go back
    assert st(layers(3), 3, stages(0, 0, 1), 128, 1, C.BF16, 66, None) == 4    # misaligned sync words
    assert st(layers(3), 3, stages(0, 0, 1), 128, 0, C.BF16, 64, None) == 0    # B == 0
    # stages rise by at most one per layer from 0, so every accepted stage map fits the limit
    assert s_max >= n_max


def test_direct_update_validation(lib):
    """DL's own AdamW step: shape, hyper-parameter and alignment rules."""
    du = lib.catq_direct_adamw_step
    hp = C.adamw()
    args = [8, 16, 16, 16, 16, 16, ctypes.byref(hp), 1, 1e-3, None]
    assert du(-1, *args[1:]) == 2
    assert du(0, None, None, None, None, None, None, 1, 1e-3, None) == 0
    assert du(*args[:6], None, *args[7:]) == 1                 # no hyper-parameters
    assert du(*args[:7], 0, *args[8:]) == 1                    # t starts at 1
    assert du(*args[:8], float("nan"), None) == 1
    assert du(*args[:8], -1e-3, None) == 1
    for bad in (C.adamw(beta1=1.0), C.adamw(beta2=-0.1), C.adamw(eps=0.0), C.adamw(weight_decay=-1.0),
                C.adamw(margin=0.5)):
        assert du(*args[:6], ctypes.byref(bad), *args[7:]) == 1
    assert du(8, 16, 16, 16, 18, 16, ctypes.byref(hp), 1, 1e-3, None) == 4
