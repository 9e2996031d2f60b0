"""Seeded synthetic calibration workloads (inputs only, no CAT-Q arithmetic).

The paper calibrates on 512 C4 sequences of 2048 tokens through Qwen3 / Llama linears
(§3.1, App. B.1).  Neither the corpus nor the checkpoints are available here, so these
generators stand in for them with the shapes of those layers and the value distributions
stated per workload below.  Every tensor comes from its own numpy sub-stream keyed by
(seed, tensor name), so any subset can be regenerated bit-identically on any machine.
Weights and activations are rounded to bf16 (round to nearest even) for the bf16
workloads; both the CUDA path and the CPU oracle read exactly those values.
"""
from __future__ import annotations

import dataclasses
import zlib

import numpy as np

# --------------------------------------------------------------------------- dtypes


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float values to bf16 (nearest, ties to even); returns the uint16 bit pattern."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact float32 value of bf16 bit patterns."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """float32 array holding the bf16-rounded values of x."""
    return bf16_to_f32(bf16_bits(x))


# --------------------------------------------------------------------------- streams


def rng(seed: int, name: str) -> np.random.Generator:
    """Independent generator for one named tensor of one seeded workload."""
    return np.random.default_rng(np.random.SeedSequence([int(seed), zlib.crc32(name.encode())]))


# --------------------------------------------------------------------------- workloads


@dataclasses.dataclass(frozen=True)
class Linear:
    name: str
    K: int  # in_features
    N: int  # out_features
    x: str  # name of the activation tensor feeding it


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    dtype: str  # "f32" or "bf16"
    M: int  # calibration tokens per step (batch x sequence length)
    g: int  # group size
    thr_init: int  # 0 = Delta0 0.5, 1 = TWN 0.7 rule
    w_std: float
    x_kind: str  # "normal", "student_t4"
    x_outlier_frac: float  # fraction of input channels scaled as outliers (activations)
    x_outlier_scale: float
    w_outlier_cols: int  # input channels of W scaled as outliers (c1)
    w_outlier_scale: float
    linears: tuple
    experts: int = 0  # > 0: MoE layer, `linears` describe one expert
    top_k: int = 0
    zipf_a: float = 0.0
    tokens: int = 0  # MoE: tokens before routing

    def linear(self, name: str) -> Linear:
        for lin in self.linears:
            if lin.name == name:
                return lin
        raise KeyError(name)

    @property
    def flops_per_step(self) -> float:
        """Algorithmic flops of fwd + dX + dW: 6 M N K per linear (per expert row for MoE)."""
        if self.experts:
            rows = self.tokens * self.top_k
            return float(sum(6.0 * rows * lin.N * lin.K for lin in self.linears))
        return float(sum(6.0 * self.M * lin.N * lin.K for lin in self.linears))


def _block(h: int, kv: int, inter: int):
    return (
        Linear("q_proj", h, h, "x_hidden"),
        Linear("k_proj", h, kv, "x_hidden"),
        Linear("v_proj", h, kv, "x_hidden"),
        Linear("o_proj", h, h, "x_attn"),
        Linear("gate_proj", h, inter, "x_hidden"),
        Linear("up_proj", h, inter, "x_hidden"),
        Linear("down_proj", inter, h, "x_ffn"),
    )


WORKLOADS = {
    # Single fp32 linear: W 512x512 ~ N(0, 0.02^2) with 4 input channels x20, X = 8 x 128
    # tokens ~ N(0, 1); channel-wise groups with the TWN 0.7 threshold rule.
    "c1_fp32_linear_512": Workload(
        name="c1_fp32_linear_512", dtype="f32", M=8 * 128, g=512, thr_init=1, w_std=0.02,
        x_kind="normal", x_outlier_frac=0.0, x_outlier_scale=1.0, w_outlier_cols=4,
        w_outlier_scale=20.0, linears=(Linear("linear", 512, 512, "x"),)),
    # Qwen3-1.7B-shaped block, 4 x 2048 tokens, 1% of channels x30.
    "c2_qwen3_1p7b_block": Workload(
        name="c2_qwen3_1p7b_block", dtype="bf16", M=4 * 2048, g=128, thr_init=0, w_std=0.02,
        x_kind="normal", x_outlier_frac=0.01, x_outlier_scale=30.0, w_outlier_cols=0,
        w_outlier_scale=1.0, linears=_block(2048, 1024, 6144)),
    # Llama-3-8B-shaped block, 4 x 2048 tokens, Student-t(4) activations.
    "c3_llama3_8b_block": Workload(
        name="c3_llama3_8b_block", dtype="bf16", M=4 * 2048, g=128, thr_init=0, w_std=0.015,
        x_kind="student_t4", x_outlier_frac=0.0, x_outlier_scale=1.0, w_outlier_cols=0,
        w_outlier_scale=1.0, linears=_block(4096, 1024, 14336)),
    # Qwen3-14B-shaped block, 2 x 2048 tokens, 0.5% of channels x50.
    "c4_qwen3_14b_block": Workload(
        name="c4_qwen3_14b_block", dtype="bf16", M=2 * 2048, g=128, thr_init=0, w_std=0.02,
        x_kind="normal", x_outlier_frac=0.005, x_outlier_scale=50.0, w_outlier_cols=0,
        w_outlier_scale=1.0, linears=_block(5120, 1024, 17408)),
    # Qwen3-235B-A22B-shaped MoE layer: 128 experts, top-8 of Zipf(1.1), 4 x 2048 tokens.
    "c5_qwen3_235b_moe": Workload(
        name="c5_qwen3_235b_moe", dtype="bf16", M=0, g=128, thr_init=0, w_std=0.02,
        x_kind="normal", x_outlier_frac=0.0, x_outlier_scale=1.0, w_outlier_cols=0,
        w_outlier_scale=1.0,
        linears=(Linear("gate_proj", 4096, 1536, "x_hidden"),
                 Linear("up_proj", 4096, 1536, "x_hidden"),
                 Linear("down_proj", 1536, 4096, "x_ffn")),
        experts=128, top_k=8, zipf_a=1.1, tokens=4 * 2048),
}


def weight(wl: Workload, lin: Linear, seed: int = 0, expert: int | None = None) -> np.ndarray:
    """float32 weight [N, K] of one linear (bf16-rounded for bf16 workloads)."""
    key = f"{wl.name}/{lin.name}/W" + ("" if expert is None else f"/e{expert}")
    r = rng(seed, key)
    W = r.standard_normal((lin.N, lin.K), dtype=np.float32) * np.float32(wl.w_std)
    if wl.w_outlier_cols:
        cols = rng(seed, key + "/outlier_cols").choice(lin.K, wl.w_outlier_cols, replace=False)
        W[:, cols] *= np.float32(wl.w_outlier_scale)
    return round_bf16(W) if wl.dtype == "bf16" else W


def activations(wl: Workload, x_name: str, M: int, K: int, seed: int = 0,
                rows: np.ndarray | None = None) -> np.ndarray:
    """float32 activations [M, K] (bf16-rounded for bf16 workloads).

    Rows are generated in blocks of 256 from per-block sub-streams, so any subset of rows
    (``rows``) can be regenerated without producing the rest.
    """
    key = f"{wl.name}/{x_name}/X/K{K}"
    cols = None
    if wl.x_outlier_frac > 0:
        n_out = max(1, int(round(wl.x_outlier_frac * K)))
        cols = rng(seed, key + "/outlier_cols").choice(K, n_out, replace=False)
    want = np.arange(M) if rows is None else np.asarray(rows)
    out = np.empty((want.size, K), dtype=np.float32)
    blocks = np.unique(want // 256)
    for b in blocks:
        r = rng(seed, f"{key}/rows{b}")
        n = min(256, M - b * 256)
        if wl.x_kind == "normal":
            blk = r.standard_normal((n, K), dtype=np.float32)
        elif wl.x_kind == "student_t4":
            blk = r.standard_t(4.0, size=(n, K)).astype(np.float32)
        else:
            raise ValueError(wl.x_kind)
        if cols is not None:
            blk[:, cols] *= np.float32(wl.x_outlier_scale)
        sel = np.nonzero(want // 256 == b)[0]
        out[sel] = blk[want[sel] - b * 256]
    return round_bf16(out) if wl.dtype == "bf16" else out


def factors(G: int, seed: int, tag: str, perturbed: bool):
    """Learnable factors (d_mu, d_alpha, d_delta), float32 [G] each.  Identity (0, 1, 1)
    is the start of calibration (§2.2); the perturbed draw (d_mu ~ U(-0.1, 0.1),
    d_alpha, d_delta ~ U(0.8, 1.2)) exercises every gradient term."""
    if not perturbed:
        return (np.zeros(G, np.float32), np.ones(G, np.float32), np.ones(G, np.float32))
    r = rng(seed, tag + "/factors")
    return (r.uniform(-0.1, 0.1, G).astype(np.float32),
            r.uniform(0.8, 1.2, G).astype(np.float32),
            r.uniform(0.8, 1.2, G).astype(np.float32))


def gradients(G: int, seed: int, tag: str):
    """Stand-ins for the three factor gradients, float32 [G] each: signed normal values whose
    scales spread log-uniformly over 1e-6 .. 1e-2, as per-group sums of a calibration
    batch do, with a few exact zeros."""
    r = rng(seed, tag + "/grads")
    out = []
    for _ in range(3):
        v = r.standard_normal(G) * 10.0 ** r.uniform(-6, -2, G)
        v[r.random(G) < 0.01] = 0.0
        out.append(v.astype(np.float32))
    return tuple(out)


def moe_routing(wl: Workload, seed: int = 0):
    """Top-k expert assignment per token: k distinct experts drawn without replacement
    (Gumbel top-k) from p_e proportional to (e + 1)^-a.  Returns (token_of_row,
    expert_row_offsets [E + 1]) for the expert-sorted row order."""
    E, T, k = wl.experts, wl.tokens, wl.top_k
    logp = -wl.zipf_a * np.log(np.arange(1, E + 1, dtype=np.float64))
    gumbel = rng(seed, f"{wl.name}/routing").gumbel(size=(T, E))
    choice = np.argsort(-(logp[None, :] + gumbel), axis=1)[:, :k]
    expert = choice.reshape(-1)
    token = np.repeat(np.arange(T), k)
    order = np.argsort(expert, kind="stable")
    counts = np.bincount(expert, minlength=E)
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)
    return token[order].astype(np.int64), offsets
