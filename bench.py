#!/usr/bin/env python
"""Throughput of the CAT-Q soft-ternary calibration step on GB300.

One step = one pass of the whole hot path over one calibration batch for every linear of
a decoder block (default: the Llama-3-8B-shaped block, 4 x 2048 tokens):
  group statistics (Eq. 3) -> fused soft-ternary forward Y = X Wq^T (Eq. 5/6, s = 30)
  -> reconstruction loss and dY against the cached teacher output (Eq. 7)
  -> dX = dY Wq -> factor gradients from dY^T X (chain rule of Eq. 3/5/6)
  -> AdamW update of the factors -> hard ternarization + 2-bit pack (Eq. 2/4).
The forward and the loss run as two calls: the fused call (catq_soft_ternary_linear_fwd_loss)
is exact but slower on this GPU (its epilogue lengthens the accumulator drain).
The metric is the algorithmic 6 M N K flops per linear (fwd + dX + dW) per second.

Prints ONE JSON line (rank 0).  `--impl reference` times the fp64 CPU oracle instead (the
only other place this file runs the oracle besides the cpu_baseline leg).
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2606_26650_gb300 import synthetic as syn  # noqa: E402

METRIC = "soft-ternary linear fwd+bwd TFLOP/s per calibration step; % of GB300 BF16 peak"
UNIT = "TFLOP/s"
DEFAULT_WORKLOAD = "c3_llama3_8b_block"
CPU_SAMPLE_LINEARS = ("q_proj", "k_proj", "down_proj")  # cpu_baseline leg of our arm
CPU_SAMPLE_ROWS = 256
REF_STEP_LINEARS = ("k_proj",)  # one step of the reference arm (runs K + W times)
# App. B.1: AdamW on the factors at learning rate 1e-3, decayed linearly to zero over 60
# epochs of ceil(512 / 3) batches of three 2048-token samples.
LR0 = 1e-3
UPDATES = 60 * -(-512 // 3)

# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) per launch, mean over the
# seven linears of the 8B-shaped block step, each captured alone (bench.py --linear NAME, the
# SOFT forward, dX and dW launches of the warm-up step; profiles/traffic_c3_linears.md); keyed
# by the hash of the kernel sources it was taken at and reported only while they are unchanged.
TRAFFIC = {"sha": "52e1c32f8e79fffe", "workload": "c3_llama3_8b_block",
           "fwd": 389121609, "dx": 416342235, "dw": 467406629}


def parse(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=60)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(syn.WORKLOADS))
    p.add_argument("--s", type=float, default=30.0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-also", action="store_true", help="skip the secondary workloads and phase")
    p.add_argument("--streams", type=int, default=4,
                   help="CUDA streams the block's linears are spread over (independent problems)")
    p.add_argument("--only", default=None,
                   choices=["moe", "decode_b1", "decode_b8", "decode_b1_staged", "block_window"],
                   help="run one secondary measurement alone and print its result (for profiling)")
    p.add_argument("--moe-experts", type=int, default=None,
                   help="with --only moe: fewer experts (same shape and routing law; for profiling)")
    p.add_argument("--linear", default=None,
                   help="run only this linear of the block (single-kernel profiling of one layer)")
    return p.parse_args(argv)


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def kernel_sources_sha() -> str:
    h = hashlib.sha256()
    for f in ("tc_gemm.cu", "catq_math.cuh", "ptx_sm100.cuh"):
        with open(os.path.join(ROOT, "paper_2606_26650_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        return dict(bf16=float(d["bf16_tflops"]), bf16_sus=float(d["bf16_tflops_sustained"]),
                    hbm=float(d["hbm_gbs"]), source="measured")
    except Exception:
        return dict(bf16=1900.0, bf16_sus=1700.0, hbm=6800.0, source="fallback")


# ------------------------------------------------------------------ CPU oracle (baseline)

def oracle_sample(wl, s, rows=CPU_SAMPLE_ROWS, linears=CPU_SAMPLE_LINEARS):
    """Times the fp64 oracle on a bounded sample of the workload: the named linears at
    `rows` tokens, every hot-path row (stats, fwd, loss, dX, factor gradients, factor
    update, pack).
    Returns (seconds, algorithmic flops)."""
    from oracle import catq_oracle as O
    total_t, flops = 0.0, 0.0
    for name in linears:
        lin = wl.linear(name)
        W = syn.weight(wl, lin).astype(np.float64)
        X = syn.activations(wl, lin.x, rows, lin.K).astype(np.float64)
        G = lin.N * lin.K // wl.g
        fac = syn.factors(G, 0, f"bench/{name}", perturbed=True)
        Y_ref = O.linear_fwd(X, W)  # cached teacher, not timed
        t0 = time.perf_counter()
        stats = O.group_stats(W, wl.g, wl.thr_init)
        Wq = O.ternary_weight(W, wl.g, stats, fac, O.PHASE_SOFT, s)[0]
        Y = O.linear_fwd(X, Wq)
        _, dY = O.recon_loss(Y, Y_ref)
        grads = O.linear_bwd(X, dY, W, wl.g, stats, fac, O.PHASE_SOFT, s)[1:]
        fac, _ = O.factor_update(fac, grads, (np.zeros(G),) * 6, 1, LR0)
        T, _, _ = O.hard_codes(W, wl.g, stats, fac)
        O.pack_codes(T)
        total_t += time.perf_counter() - t0
        flops += 6.0 * rows * lin.N * lin.K
    return total_t, flops


def max_over_ranks(ms: float, world: int, device) -> float:
    """The slowest rank's step time, on every rank (the timing rule: max over ranks)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(flops_per_rank_step: float, ms: float, world: int) -> float:
    """Whole-job TFLOP/s: every rank runs the same step on its own inputs (weak scaling), so
    the job does `world` times one rank's work in the slowest rank's time."""
    return world * flops_per_rank_step / (ms * 1e-3) / 1e12


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def sample_text(wl, rows=CPU_SAMPLE_ROWS, linears=CPU_SAMPLE_LINEARS):
    return (f"{'+'.join(linears)} of {wl.name} at {rows} of {wl.M} tokens, fp64 numpy oracle, all hot-path rows "
            f"(stats, fwd, loss, dX, factor grads, AdamW factor update, pack); matmuls on multi-threaded BLAS, "
            f"elementwise single-threaded; per-layer modulation cost is paid once per sample, as in the full step")


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return
    wl = syn.WORKLOADS[args.workload]
    for _ in range(args.warmup):
        oracle_sample(wl, args.s, linears=REF_STEP_LINEARS)
    times, flops = [], 0.0
    for _ in range(args.steps):
        t, flops = oracle_sample(wl, args.s, linears=REF_STEP_LINEARS)
        times.append(t)
    tot = sum(times)
    value = flops * len(times) / tot / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(wl, args),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                         "sample": sample_text(wl, linears=REF_STEP_LINEARS) + "; one sample per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def workload_config(wl, args):
    return {"workload": wl.name + (f"/{args.linear}" if getattr(args, "linear", None) else ""), "tokens": wl.M,
            "group_size": wl.g, "phase": "soft", "s": args.s,
            "linears": {lin.name: [lin.K, lin.N] for lin in wl.linears},
            "flops_per_step": wl.flops_per_step, "streams": getattr(args, "streams", 1),
            "l2": "inputs larger than L2 (per-step working set of weights and activations > 129 MB)"}


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ GPU arm

KINDS = ("fwd", "dx", "dw")
# Block workloads also timed (secondary lines of the JSON output): the Qwen3-14B-shaped block
# the 60%-of-peak target also names, and the Qwen3-1.7B-shaped one.
ALSO_WORKLOADS = ("c4_qwen3_14b_block", "c2_qwen3_1p7b_block")


class FactorUpdate:
    """The optimizer step closing each calibration step: AdamW on every linear's three
    factors (moments zero at the start) at the linearly decayed learning rate of the update
    count.  After a full calibration's UPDATES updates a fresh calibration starts: the
    count returns to 1 and the moments to zero (never reached by the default run)."""

    def __init__(self, C, torch, dev, group_counts):
        self.C, self.hp, self.t, self.lr = C, C.adamw(), 0, LR0
        # zeros copied from the host: no fill kernel among the step's launches
        self.moments = [torch.zeros(6 * G).to(dev) for G in group_counts]

    def advance(self):
        if self.t == UPDATES:
            self.t = 0
            for m in self.moments:
                m.zero_()
        self.t += 1
        self.lr = self.C.catq_linear_decay_lr(LR0, self.t - 1, UPDATES)

    def apply(self, i, layer, grads):
        self.C.catq_factor_adamw_step(layer.d_mu, layer.d_alpha, layer.d_delta, *grads, self.moments[i], self.hp,
                                      self.t, self.lr)


class BlockRun:
    """Device state and one calibration step of a block workload: every linear's seeded
    inputs, layer and teacher output, and per-stream workspaces.

    The block's linears are independent calibration problems (one loss per linear output,
    Eq. 7), so a step spreads them over `nstreams` CUDA streams: one linear's kernels can
    start on the SMs another linear's last tile wave leaves idle.  A step forks from and
    joins back into the current stream."""

    def __init__(self, C, torch, wl, dev, rank, nstreams, recon=0):
        self.C, self.torch, self.wl = C, torch, wl
        M = self.M = wl.M
        bf = torch.bfloat16 if wl.dtype == "bf16" else torch.float32

        def upload(a):
            if wl.dtype == "bf16":
                return torch.from_numpy(syn.bf16_bits(a).view(np.int16)).to(dev).view(torch.bfloat16)
            return torch.from_numpy(a).to(dev)

        Xs = {}
        for lin in wl.linears:
            if (lin.x, lin.K) not in Xs:
                Xs[(lin.x, lin.K)] = upload(syn.activations(wl, lin.x, M, lin.K, seed=rank))
        self.st = []
        ws_bwd = ws_loss = 0
        for lin in wl.linears:
            G = lin.N * lin.K // wl.g
            fac = [torch.from_numpy(f).to(dev) for f in syn.factors(G, rank, f"bench/{lin.name}", perturbed=True)]
            layer = C.Layer.create(upload(syn.weight(wl, lin, seed=rank)), wl.g, *fac, recon=recon)
            C.catq_group_stats(layer, wl.thr_init)
            d = dict(lin=lin, layer=layer, X=Xs[(lin.x, lin.K)],
                     Yt=torch.empty(M, lin.N, dtype=bf, device=dev), Y=torch.empty(M, lin.N, dtype=bf, device=dev),
                     dY=torch.empty(M, lin.N, dtype=bf, device=dev), dX=torch.empty(M, lin.K, dtype=bf, device=dev),
                     grads=[torch.empty(G, device=dev) for _ in range(3)],
                     codes=torch.empty(lin.N * lin.K // 4, dtype=torch.uint8, device=dev),
                     alpha=torch.empty(G, device=dev), loss=torch.empty(1, device=dev))
            C.catq_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), d["X"], d["Yt"])
            ws_bwd = max(ws_bwd, C.catq_bwd_workspace_bytes(layer, M))
            ws_loss = max(ws_loss, C.catq_recon_loss_workspace_bytes(M * lin.N))
            self.st.append(d)
        self.upd = FactorUpdate(C, torch, dev, [d["grads"][0].numel() for d in self.st])
        self.main = torch.cuda.current_stream()
        self.lanes = [self.main] if nstreams == 1 else [torch.cuda.Stream(device=dev) for _ in range(nstreams)]
        self.wsbs = [C.workspace(ws_bwd, dev) for _ in self.lanes]
        self.wsls = [C.workspace(ws_loss, dev) for _ in self.lanes]
        torch.cuda.synchronize()

    def step(self, sched, ev=None, serial=False, before=None, after=None):
        """One step at schedule point `sched`; `serial` runs every linear on the current
        stream (kernel timing); before(i) / after(i) run on linear i's stream around its
        kernels (e2e copies); ev[i][kind] are (start, end) events around each GEMM call."""
        C, torch, wl = self.C, self.torch, self.wl
        use = [self.main] if serial else self.lanes
        self.upd.advance()
        if len(use) > 1:
            fork = torch.cuda.Event()
            fork.record(self.main)
            for s in use:
                s.wait_event(fork)
        for i, d in enumerate(self.st):
            k = i % len(use)
            with torch.cuda.stream(use[k]):
                if before is not None:
                    before(i)
                L = d["layer"]
                C.catq_group_stats(L, wl.thr_init)
                if ev is not None:
                    ev[i]["fwd"][0].record()
                C.catq_soft_ternary_linear_fwd(L, sched, d["X"], d["Y"])
                if ev is not None:
                    ev[i]["fwd"][1].record()
                C.catq_recon_loss(d["Y"], d["Yt"], d["loss"], d["dY"], self.wsls[k])
                if ev is not None:
                    ev[i]["dx"][0].record()
                C.catq_soft_ternary_linear_bwd(L, sched, d["X"], d["dY"], dX=d["dX"])
                if ev is not None:
                    ev[i]["dx"][1].record()
                    ev[i]["dw"][0].record()
                C.catq_soft_ternary_linear_bwd(L, sched, d["X"], d["dY"], None, *d["grads"], workspace=self.wsbs[k])
                if ev is not None:
                    ev[i]["dw"][1].record()
                self.upd.apply(i, L, d["grads"])
                C.catq_hard_ternarize_pack(L, d["codes"], d["alpha"])
                if after is not None:
                    after(i)
        if len(use) > 1:
            for s in use:
                join = torch.cuda.Event()
                join.record(s)
                self.main.wait_event(join)

    def ms_per_step(self, sched, steps, warmup, barrier):
        """Mean step time over `steps` steps after `warmup`, CUDA events on this stream."""
        torch = self.torch
        for _ in range(warmup):
            self.step(sched)
        barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            self.step(sched)
        b.record()
        barrier()
        status = self.C.catq_device_status()
        if status != 0:
            raise SystemExit(f"device status {self.C.STATUS.get(status, status)} in a secondary timed region")
        return a.elapsed_time(b) / steps


def run_ours(args):
    import torch

    from paper_2606_26650_gb300 import catq as C

    rank, local, world = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    wl = syn.WORKLOADS[args.workload]
    if wl.experts:
        raise SystemExit("MoE workloads are parity cases, not bench lines")
    if args.linear:
        wl = dataclasses.replace(wl, linears=(wl.linear(args.linear),))
    sched = C.schedule(C.PHASE_SOFT, args.s)
    nstreams = max(1, args.streams)
    blk = BlockRun(C, torch, wl, dev, rank, nstreams)
    st, M = blk.st, blk.M
    kinds = KINDS

    def step(ev=None, serial=False, before=None, after=None):
        blk.step(sched, ev, serial, before, after)

    # per linear: stats; operand constants + forward; loss (partial + final); operand
    # constants + dX; dW + gradient reduce; factor update; pack
    launches_per_step = len(st) * (1 + 2 + 2 + 2 + 2 + 1 + 1)

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
            torch.cuda.synchronize()

    for _ in range(args.warmup):
        step()
    barrier()
    status = C.catq_device_status()
    if status != 0:
        raise SystemExit(f"device status {C.STATUS.get(status, status)} during warm-up")

    E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    evs = [[{k: (E(), E()) for k in kinds} for _ in st] for _ in range(args.steps)]
    t_start, t_end = E(), E()
    # With one stream the step's own timed region also times each kernel.  With several,
    # kernels of different linears share the GPU, so a second timed region of the same K
    # steps on one stream times each kernel on its own for the roofline.
    with ClockSampler(local) as clk:
        barrier()
        t_start.record()
        for k in range(args.steps):
            step(evs[k] if nstreams == 1 else None)
        t_end.record()
        barrier()
    status = C.catq_device_status()
    if status != 0:
        raise SystemExit(f"device status {C.STATUS.get(status, status)} in the timed region")
    ms = max_over_ranks(t_start.elapsed_time(t_end) / args.steps, world, dev)
    flops_step = wl.flops_per_step
    value = job_throughput(flops_step, ms, world)
    if nstreams > 1:
        barrier()
        for k in range(args.steps):
            step(evs[k], serial=True)
        barrier()
        if C.catq_device_status() != 0:
            raise SystemExit("device status set in the kernel-timing region")

    # per-kernel live timing (CUDA events on the launching stream)
    per = {k: 0.0 for k in kinds}
    for k in range(args.steps):
        for i in range(len(st)):
            for kind in kinds:
                a, b = evs[k][i][kind]
                per[kind] += a.elapsed_time(b)
    flops_kind = sum(2.0 * M * d["lin"].N * d["lin"].K for d in st) * args.steps
    dom = max(kinds, key=lambda k: per[k])
    peaks = measured_peaks()
    achieved = flops_kind / (per[dom] * 1e-3) / 1e12
    kernel_name = {"fwd": "fused_gemm_kernel (forward, K-major Wq operand)",
                   "dx": "fused_gemm_kernel (dX, MN-major Wq operand)",
                   "dw": "dw_kernel + grad_reduce_kernel (dW factor-gradient epilogue)"}[dom]
    sha = kernel_sources_sha()
    traffic = (TRAFFIC.get(dom) if TRAFFIC.get("sha") == sha and TRAFFIC.get("workload") == wl.name
               else None)
    esz = 2 if wl.dtype == "bf16" else 4
    # forward: X, W, Y; dX: dY, W, dX; dW: dY, X, W (plus the per-group arrays)
    algo_bytes = sum(esz * (M * d["lin"].K + d["lin"].N * d["lin"].K + M * d["lin"].N)
                     + 4 * (d["lin"].N * d["lin"].K // wl.g) * (9 if dom == "dw" else 6) for d in st) / len(st)
    # The per-kernel durations come from a region of `steps` steps on one stream (a fraction
    # of a second at the default 60 steps), not from a seconds-long loop under the power cap,
    # so the burst peak is the denominator; the sustained fraction is reported beside it.
    roofline = {"bound": "tensor", "kernel": kernel_name, "achieved": achieved, "peak": peaks["bf16"],
                "unit": UNIT, "frac": achieved / peaks["bf16"], "traffic": traffic,
                "traffic_algorithmic": algo_bytes,
                "peak_kind": f"bf16 dense burst ({peaks['source']})",
                "frac_of_sustained": achieved / peaks["bf16_sus"],
                "per_kernel_ms_per_step": {k: per[k] / args.steps for k in kinds},
                "kernel_timing": ("the step's timed region (one stream)" if nstreams == 1 else
                                  f"one stream, {args.steps} steps right after the step's timed region "
                                  f"(the step itself spreads the linears over {nstreams} streams)"),
                "per_kernel_tflops": {k: flops_kind / (per[k] * 1e-3) / 1e12 for k in kinds}}

    e2e = None
    if not args.no_e2e:
        e2e = measure_e2e(args, C, torch, st, step, barrier, flops_step, world, dev)

    # Secondary measurements (same code path, fewer steps): the HARD phase of this workload,
    # and the other block workloads the 60%-of-peak target names or that fit the same step.
    also = {}
    if not args.no_also:
        n2, w2 = max(5, args.steps // 4), 3

        def entry(wl2, ms2):
            ms2 = max_over_ranks(ms2, world, dev)
            v2 = job_throughput(wl2.flops_per_step, ms2, world)
            return {"value": v2, "ms_per_step": ms2, "frac_of_burst": v2 / world / peaks["bf16"], "steps": n2}

        hard = blk.ms_per_step(C.schedule(C.PHASE_HARD, args.s), n2, w2, barrier)
        also[f"{wl.name}/hard"] = dict(entry(wl, hard), phase="hard", s=args.s)
        del blk, st, step
        torch.cuda.empty_cache()
        # the W ~ alpha T + mu reconstruction (the tab:mu variant) on the same workload
        bmu = BlockRun(C, torch, wl, dev, rank, nstreams, recon=C.RECON_ALPHA_T_MU)
        also[f"{wl.name}/soft_mu"] = dict(entry(wl, bmu.ms_per_step(sched, n2, w2, barrier)), phase="soft", s=args.s,
                                          recon="alpha_T_plus_mu")
        del bmu
        torch.cuda.empty_cache()
        also[f"{wl.name}/decode_b1"] = measure_decode(C, torch, wl, dev, peaks, rows=1)
        also[f"{wl.name}/decode_b8"] = measure_decode(C, torch, wl, dev, peaks, rows=8)
        also[f"{wl.name}/decode_b1_mu"] = measure_decode(C, torch, wl, dev, peaks, rows=1, with_mu=True)
        also[f"{wl.name}/decode_b1_staged"] = measure_decode(C, torch, wl, dev, peaks, rows=1, staged=True)
        also["c5_qwen3_235b_moe/soft"] = measure_moe(C, torch, dev, peaks, world, args.s)
        also[f"{wl.name}/fig_error_k_proj"] = measure_fig_error(C, torch, wl, dev, args.s)
        if wl.name in BLOCK_WINDOW_SHAPES and not args.linear:
            also[f"{wl.name}/block_window"] = measure_block_window(C, torch, wl, dev, peaks, world, args.s, barrier,
                                                                   streams=nstreams)
        for name in ALSO_WORKLOADS:
            if name == wl.name:
                continue
            wl2 = syn.WORKLOADS[name]
            b2 = BlockRun(C, torch, wl2, dev, rank, nstreams)
            also[f"{name}/soft"] = dict(entry(wl2, b2.ms_per_step(sched, n2, w2, barrier)), phase="soft", s=args.s)
            del b2
            torch.cuda.empty_cache()
            if name in BLOCK_WINDOW_SHAPES and not args.linear:
                also[f"{name}/block_window"] = measure_block_window(C, torch, wl2, dev, peaks, world, args.s, barrier,
                                                                    streams=nstreams)

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        t, fl = oracle_sample(wl, args.s)
        cpu = {"value": fl / t / 1e12, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": sample_text(wl), "seconds": t}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
            "config": workload_config(wl, args),
            "frac_of_bf16_peak": {"sustained": value / world / peaks["bf16_sus"],
                                  "burst": value / world / peaks["bf16"], "source": peaks["source"]},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": launches_per_step * args.steps, "clocks": clk.summary(),
            "also": also,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


# Decoder blocks of the block-window lines: (hidden, query heads, key/value heads, head dim,
# MLP width, sequences, tokens per sequence, RoPE base, per-head query/key norm).  The Llama-3-8B
# block has no query/key norm; the Qwen3 blocks normalise every query and key head.
BLOCK_WINDOW_SHAPES = {
    "c3_llama3_8b_block": (4096, 32, 8, 128, 14336, 4, 2048, 500000.0, False),
    "c4_qwen3_14b_block": (5120, 40, 8, 128, 17408, 2, 2048, 1000000.0, True),
    "c2_qwen3_1p7b_block": (2048, 16, 8, 128, 6144, 4, 2048, 1000000.0, True),
}


def measure_block_window(C, torch, wl, dev, peaks, world, s, barrier, steps=5, warmup=3, streams=4):
    """Eq. 7 over a window of one whole decoder block (§2.4) of the workload's shape (e.g. the
    Llama-3-8B block: 4 x 2048 tokens, 32 query heads and 8 key/value heads of 128, RoPE base
    500000).  One step is the student block forward (seven soft-ternary linears, RMSNorm,
    rotary embedding, causal attention, SwiGLU; the Qwen3 blocks' query/key head norms), the
    loss on the block output against the cached teacher output, the block backward into every
    linear's factor gradients, and the AdamW update of all factors.  Throughput counts the
    linears' 6 T N K and attention's 7 B h S^2 d flops; the attention forward + backward is also
    timed alone on the same tensors.  `streams`: the block's main stream and streams - 1 side
    streams for its independent calls."""
    from paper_2606_26650_gb300 import block as BK
    H, nh, nkv, d, I, B, S, base, qk_norm = BLOCK_WINDOW_SHAPES[wl.name]
    shape = BK.BlockShape(H=H, n_heads=nh, n_kv_heads=nkv, d=d, I=I, B=B, S=S, base=base, eps=1e-5)
    assert shape.T == wl.M
    bf = torch.bfloat16

    def upload(a):
        return torch.from_numpy(syn.bf16_bits(a).view(np.int16)).to(dev).view(bf)

    W = {lin.name: upload(syn.weight(wl, lin)) for lin in wl.linears}
    r = syn.rng(97, "bench/block_window")
    g1, g2 = (torch.from_numpy(r.uniform(0.5, 1.5, shape.H).astype(np.float32)).to(dev) for _ in range(2))
    fac = {n: tuple(torch.from_numpy(f).to(dev) for f in syn.factors(W[n].numel() // wl.g, 0, f"window/{n}", True))
           for n in W}
    norms = {}
    if qk_norm:
        norms = {k: torch.from_numpy(r.uniform(0.5, 1.5, d).astype(np.float32)).to(dev) for k in ("q_norm", "k_norm")}
    blk = BK.Block(shape, W, g1, g2, wl.g, factors=fac, side_streams=max(0, streams - 1), **norms)
    x = upload(syn.activations(wl, "x_hidden", shape.T, shape.H))
    out_ref = torch.empty(shape.T, shape.H, dtype=torch.float32, device=dev)
    blk.teacher(x, out_ref)
    loss = torch.zeros(1, dtype=torch.float32, device=dev)
    grads = {n: [torch.empty(W[n].numel() // wl.g, dtype=torch.float32, device=dev) for _ in range(3)] for n in W}
    upd = FactorUpdate(C, torch, dev, [W[n].numel() // wl.g for n in BK.LINEARS])
    sched = C.schedule(C.PHASE_SOFT, s)

    def step():
        blk.step(x, out_ref, sched, loss, grads)
        upd.advance()
        for i, n in enumerate(BK.LINEARS):
            upd.apply(i, blk.layers[n], grads[n])

    def timed(fn, n, w):
        for _ in range(w):
            fn()
        barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(n):
            fn()
        b.record()
        barrier()
        status = C.catq_device_status()
        if status != 0:
            raise SystemExit(f"device status {C.STATUS.get(status, status)} in the block-window timed region")
        return a.elapsed_time(b) / n

    ms = max_over_ranks(timed(step, steps, warmup), world, dev)
    first_loss = loss.item()

    def attention():
        C.catq_attention_fwd(blk.q, blk.k, blk.v, blk.a, blk.lse, shape.B, shape.S, shape.n_heads, shape.n_kv_heads,
                             shape.d)
        C.catq_attention_bwd(blk.q, blk.k, blk.v, blk.a, blk.da, blk.lse, blk.delta, blk.dq, blk.dk, blk.dv, shape.B,
                             shape.S, shape.n_heads, shape.n_kv_heads, shape.d)

    attn_ms = timed(attention, steps, 2)
    flops = shape.linear_flops() + shape.attention_flops()
    value = job_throughput(flops, ms, world)
    out = {"value": value, "unit": UNIT, "ms_per_step": ms, "steps": steps, "frac_of_burst": value / world / peaks["bf16"],
           "flops_per_step": {"linears": shape.linear_flops(), "attention": shape.attention_flops()},
           "attention_fwd_bwd_ms": attn_ms,
           "attention_tflops": shape.attention_flops() / (attn_ms * 1e-3) / 1e12,
           "loss_after_steps": first_loss, "phase": "soft", "s": s, "qk_norm": qk_norm, "streams": 1 + len(blk.sides),
           "shape": dataclasses.asdict(shape), "l2": "working set > L2 (no flush)"}
    del blk, W, x, out_ref, grads, upd
    torch.cuda.empty_cache()
    return out


# Linears of a decoder block that may run in one launch (their inputs do not depend on each
# other): q, k, v read the block's input; o reads the attention output; gate and up read the
# post-attention input; down reads their product.
DECODE_GROUPS = (("q_proj", "k_proj", "v_proj"), ("o_proj",), ("gate_proj", "up_proj"), ("down_proj",))


def measure_decode(C, torch, wl, dev, peaks, blocks=32, rows=1, steps=20, with_mu=False, staged=False):
    """Inference with the deployed form of every linear of `blocks` blocks shaped like `wl`,
    for `rows` token rows: one decode step reads every layer's 2-bit codes and group scales
    (and group offsets, `with_mu`) once (working set far beyond L2), layer sets in block order
    (DECODE_GROUPS: q/k/v, o, gate/up, down), as a decode step must.
    staged: the layer sets are the stages of catq_ternary_infer_staged, four blocks (28 layers,
    16 stages) per cooperative launch; otherwise one catq_ternary_infer_batched launch per set,
    captured in a CUDA graph and replayed.  value = algorithmic bytes / time."""
    import ctypes
    gen = torch.Generator(device=dev)
    gen.manual_seed(0)
    launches, nbytes, g = [], 0, wl.g
    for _ in range(blocks):
        for names in DECODE_GROUPS:
            group = []
            for name in names:
                lin = wl.linear(name)
                N, K = lin.N, lin.K
                r = torch.randint(0, 81, (N * K // 4,), generator=gen, device=dev, dtype=torch.int32)
                codes = (r % 3 + ((r // 3) % 3) * 4 + ((r // 9) % 3) * 16 + (r // 27) * 64).to(torch.uint8)
                alpha = torch.rand(N * K // g, generator=gen, device=dev) * 0.02 + 0.01
                X = torch.randn(rows, K, generator=gen, device=dev).to(torch.bfloat16)
                Y = torch.empty(rows, N, dtype=torch.bfloat16, device=dev)
                mu = (torch.rand(N * K // g, generator=gen, device=dev) - 0.5) * 0.01 if with_mu else None
                group.append((codes, alpha, N, K, X, Y, mu))
                nbytes += codes.numel() + alpha.numel() * 4 + X.numel() * 2 + Y.numel() * 2
                nbytes += 0 if mu is None else mu.numel() * 4
            launches.append(group)
    if staged:
        per_call = 4  # blocks per launch: 28 layers, 16 stages
        calls = []
        sync = torch.zeros(C.catq_ternary_infer_sync_bytes() // 4, dtype=torch.int32, device=dev)
        groups_per_call = per_call * len(DECODE_GROUPS)
        for c0 in range(0, len(launches), groups_per_call):
            layers, stages = [], []
            for si, group in enumerate(launches[c0:c0 + groups_per_call]):
                layers += group
                stages += [si] * len(group)
            arr, B = C._infer_layer_array(layers, g, "bench")
            st = (ctypes.c_int32 * len(stages))(*stages)
            calls.append((arr, len(layers), st, B))
        lib, sp = C.lib(), ctypes.c_void_p(sync.data_ptr())

        def run():
            cs = C._stream()
            for arr, n, st, B in calls:
                C._check(lib.catq_ternary_infer_staged(arr, n, st, g, B, C.BF16, sp, cs), "bench decode")
        n_launch = len(calls)
    else:
        side = torch.cuda.Stream(device=dev)
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):  # warm-up outside the capture
            for group in launches:
                C.catq_ternary_infer_batched(group, g)
        torch.cuda.current_stream().wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for group in launches:
                C.catq_ternary_infer_batched(group, g)

        def run():
            graph.replay()
        n_launch = len(launches)
    for _ in range(3):
        run()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(steps):
        run()
    b.record()
    torch.cuda.synchronize()
    status = C.catq_device_status()
    if status != 0:
        raise SystemExit(f"device status {C.STATUS.get(status, status)} in the decode timing")
    ms = a.elapsed_time(b) / steps
    gbs = nbytes / (ms * 1e-3) / 1e9
    del launches, run
    torch.cuda.empty_cache()
    return {"kernel": "ternary_mma_kernel (" + ("catq_ternary_infer_staged, cooperative" if staged else
                                               "catq_ternary_infer_batched, CUDA graph") + ")",
            "blocks": blocks, "token_rows": rows, "launches_per_step": n_launch, "bytes_per_step": nbytes,
            "us_per_step": ms * 1e3, "value": gbs, "unit": "GB/s", "peak": peaks["hbm"],
            "frac_of_hbm": gbs / peaks["hbm"], "steps": steps, "with_mu": with_mu}


def measure_fig_error(C, torch, wl, dev, s0, epochs=20, batches=3, rows=2048, lr0=1e-3):
    """The synthetic analogue of Fig. fig:error (§2.2) on the block's k_proj: per-group weight
    reconstruction error of the hard ternarization under the static absmean rule (SA), direct
    learning started from it (DL) and the learnable modulation (LM), the learned two after
    `epochs` x `batches` calibration steps of `rows` tokens with hard ternarization throughout
    (the figure's setting), AdamW at lr0 decayed linearly.  Errors are per group, relative to
    the group's mean squared weight."""
    lin = wl.linear("k_proj")
    N, K, g = lin.N, lin.K, wl.g
    G = N * K // g

    def up(a):
        return torch.from_numpy(syn.bf16_bits(a).view(np.int16)).to(dev).view(torch.bfloat16)

    W = up(syn.weight(wl, lin))
    xs = [up(syn.activations(wl, lin.x, (b + 1) * rows, K)[b * rows:]) for b in range(batches)]
    w2 = (W.float().reshape(G, g) ** 2).mean(dim=1)
    out = {}
    for kind in ("SA", "DL", "LM"):
        layer = C.Layer.create(W, g)
        C.catq_group_stats(layer, C.THR_HALF if kind == "LM" else C.THR_ABSMEAN)
        if kind != "SA":
            hp = C.adamw()
            moments = torch.zeros((6 if kind == "LM" else 4) * G, device=dev)
            grads = [torch.empty(G, device=dev) for _ in range(3)]
            loss = torch.empty(1, device=dev)
            yts = []
            for xb in xs:
                yt = torch.empty(rows, N, dtype=torch.bfloat16, device=dev)
                C.catq_soft_ternary_linear_fwd(layer, C.schedule(C.PHASE_TEACHER), xb, yt)
                yts.append(yt)
            Y, dY = torch.empty_like(yts[0]), torch.empty_like(yts[0])
            wsl = C.workspace(C.catq_recon_loss_workspace_bytes(Y.numel()), dev)
            wsb = C.workspace(C.catq_bwd_workspace_bytes(layer, rows), dev)
            sched = C.schedule(C.PHASE_HARD, s0)
            t = 0
            for _ in range(epochs):
                for xb, yt in zip(xs, yts):
                    C.catq_soft_ternary_linear_fwd(layer, sched, xb, Y)
                    C.catq_recon_loss(Y, yt, loss, dY, wsl)
                    C.catq_soft_ternary_linear_bwd(layer, sched, xb, dY, None, *grads, workspace=wsb)
                    lr = C.catq_linear_decay_lr(lr0, t, epochs * batches)
                    t += 1
                    if kind == "LM":
                        C.catq_factor_adamw_step(layer.d_mu, layer.d_alpha, layer.d_delta, *grads, moments, hp, t, lr)
                    else:
                        C.catq_direct_adamw_step(layer.d_alpha, layer.d_delta, grads[1], grads[2], moments, hp, t, lr)
        err = torch.empty(G, device=dev)
        C.catq_group_recon_error(layer, err)
        out[kind] = (err / w2).cpu().numpy().astype(np.float64)
    status = C.catq_device_status()
    if status != 0:
        raise SystemExit(f"device status {C.STATUS.get(status, status)} in the fig:error run")
    res = {k: {"mean": float(v.mean()), "median": float(np.median(v)), "p99": float(np.quantile(v, 0.99)),
               "max": float(v.max())} for k, v in out.items()}
    res["groups"] = G
    res["groups_worse_than_SA"] = {k: int((out[k] > out["SA"]).sum()) for k in ("DL", "LM")}
    res["setting"] = (f"k_proj {K}->{N}, g {g}, {epochs} epochs x {batches} batches of {rows} tokens, hard "
                      f"ternarization throughout (backward at s = {s0}), AdamW lr {lr0} decayed linearly; error = "
                      f"mean (W - Wq)^2 / mean W^2 per group")
    return res


def measure_moe(C, torch, dev, peaks, world, s, steps=5, warmup=2, experts=None, nstreams=3):
    """One calibration step of the Qwen3-235B-shaped MoE layer: gate/up/down of all 128
    experts over 8192 tokens routed top-8 (65,536 expert-sorted rows, Zipf(1.1) loads) through
    the grouped calls (stats once; per step forward, loss, backward, factor update, pack).  Weights and
    activations are drawn on the device (seeded); value = sum 6 M_e N K / step time.
    The three linears are independent calibration problems (one loss per linear output), so a
    step spreads them over `nstreams` CUDA streams, forking from and joining back into the
    current stream.  `experts` (profiling only) keeps the expert shape and routing law with
    fewer experts and proportionally fewer tokens, so that a capture holds less device memory."""
    wl = syn.WORKLOADS["c5_qwen3_235b_moe"]
    if experts:
        wl = dataclasses.replace(wl, experts=int(experts), tokens=wl.tokens * int(experts) // wl.experts)
    token_of_row, off = syn.moe_routing(wl, seed=0)
    R, E, g = int(off[-1]), wl.experts, wl.g
    gen = torch.Generator(device=dev)
    gen.manual_seed(0)
    tok = torch.from_numpy(token_of_row).to(dev)
    xs = {"x_hidden": torch.randn(wl.tokens, 4096, generator=gen, device=dev).to(torch.bfloat16)[tok],
          "x_ffn": torch.randn(R, 1536, generator=gen, device=dev).to(torch.bfloat16)}
    sched, teacher = C.schedule(C.PHASE_SOFT, s), C.schedule(C.PHASE_TEACHER)
    lins, flops = [], 0.0
    for lin in wl.linears:
        N, K = lin.N, lin.K
        G = N * K // g
        W = (torch.randn(E * N, K, generator=gen, device=dev) * wl.w_std).to(torch.bfloat16).reshape(E, N, K)
        fac = [(torch.rand(E * G, generator=gen, device=dev) - 0.5) * 0.2,
               0.8 + 0.4 * torch.rand(E * G, generator=gen, device=dev),
               0.8 + 0.4 * torch.rand(E * G, generator=gen, device=dev)]
        layer = C.GroupedLayer.create(W, g, *fac)
        C.catq_group_stats(layer.dense, wl.thr_init)
        X = xs[lin.x]
        Yt = torch.empty(R, N, dtype=torch.bfloat16, device=dev)
        C.catq_grouped_soft_ternary_linear_fwd(layer, teacher, X, off, Yt)
        lins.append(dict(layer=layer, X=X, Yt=Yt, Y=torch.empty_like(Yt), dY=torch.empty_like(Yt),
                         dX=torch.empty_like(X), grads=[torch.empty(E * G, device=dev) for _ in range(3)],
                         codes=torch.empty(E * N * K // 4, dtype=torch.uint8, device=dev),
                         alpha=torch.empty(E * G, device=dev), loss=torch.empty(1, device=dev),
                         wsb=C.workspace(C.catq_grouped_bwd_workspace_bytes(layer, off), dev),
                         wsl=C.workspace(C.catq_recon_loss_workspace_bytes(R * N), dev)))
        flops += 6.0 * R * N * K
    upd = FactorUpdate(C, torch, dev, [d["grads"][0].numel() for d in lins])
    main = torch.cuda.current_stream()
    lanes = [main] if nstreams <= 1 else [torch.cuda.Stream(device=dev) for _ in range(nstreams)]

    def step():
        upd.advance()
        if len(lanes) > 1:
            fork = torch.cuda.Event()
            fork.record(main)
            for ln in lanes:
                ln.wait_event(fork)
        for i, d in enumerate(lins):
            with torch.cuda.stream(lanes[i % len(lanes)]):
                C.catq_grouped_soft_ternary_linear_fwd(d["layer"], sched, d["X"], off, d["Y"])
                C.catq_recon_loss(d["Y"], d["Yt"], d["loss"], d["dY"], d["wsl"])
                C.catq_grouped_soft_ternary_linear_bwd(d["layer"], sched, d["X"], d["dY"], off, d["dX"], *d["grads"],
                                                       workspace=d["wsb"])
                upd.apply(i, d["layer"].dense, d["grads"])
                C.catq_hard_ternarize_pack(d["layer"].dense, d["codes"], d["alpha"])
        if len(lanes) > 1:
            for ln in lanes:
                join = torch.cuda.Event()
                join.record(ln)
                main.wait_event(join)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index or 0) as clk:
        a.record()
        h0 = time.perf_counter()
        for _ in range(steps):
            step()
        host_ms = (time.perf_counter() - h0) * 1e3 / steps  # issuing the calls, per step
        b.record()
        torch.cuda.synchronize()
    status = C.catq_device_status()
    if status != 0:
        raise SystemExit(f"device status {C.STATUS.get(status, status)} in the MoE timing")
    ms = max_over_ranks(a.elapsed_time(b) / steps, world, dev)
    value = job_throughput(flops, ms, world)
    counts = np.diff(off)
    del lins, xs
    torch.cuda.empty_cache()
    return {"value": value, "ms_per_step": ms, "frac_of_burst": value / world / peaks["bf16"], "steps": steps,
            "experts": E, "routed_rows": R, "rows_per_expert": [int(counts.min()), int(np.median(counts)),
                                                                 int(counts.max())],
            "path": "grouped calls: one persistent launch for every expert's forward and dX tiles, grouped "
                    "factor-gradient launches of up to 64 experts",
            "streams": len(lanes),
            "phase": "soft", "s": s, "host_issue_ms_per_step": host_ms, "clocks": clk.summary()}


def measure_e2e(args, C, torch, st, step, barrier, flops_step, world, dev):
    """Same step through the public API with each step's calibration batch (activations) and
    teacher outputs copied from pinned host memory, and its losses and factor gradients read
    back.  Inputs are double-buffered on the device: a copy stream brings step t + 1's inputs
    (in linear order, one event per linear) while step t computes on the other buffer set,
    once step t - 1 is done with it; each linear of a step starts when its own inputs have
    landed, and its results go back as soon as its kernels finish.  Every step's copies lie
    inside the timed region."""
    xs_h, yts_h = {}, []
    for d in st:
        key = d["X"].data_ptr()
        if key not in xs_h:
            xs_h[key] = torch.empty(d["X"].shape, dtype=d["X"].dtype, pin_memory=True)
            xs_h[key].copy_(d["X"])
        yt = torch.empty(d["Yt"].shape, dtype=d["Yt"].dtype, pin_memory=True)
        yt.copy_(d["Yt"])
        yts_h.append(yt)
    # two device buffer sets; set 0 is the bench's own tensors
    sets = []
    for p in range(2):
        xd = {key: (d["X"] if p == 0 else torch.empty_like(d["X"])) for d in st for key in [d["X"].data_ptr()]}
        sets.append((xd, [d["Yt"] if p == 0 else torch.empty_like(d["Yt"]) for d in st]))
    keys = [d["X"].data_ptr() for d in st]
    outs = [(t, torch.empty(t.shape, dtype=t.dtype, pin_memory=True)) for d in st for t in [d["loss"]] + d["grads"]]
    h2d = sum(h.numel() * h.element_size() for h in xs_h.values()) + sum(h.numel() * h.element_size() for h in yts_h)
    d2h = sum(h.numel() * h.element_size() for _, h in outs)

    main = torch.cuda.current_stream()
    copier = torch.cuda.Stream(device=dev)
    out_of = [[(t, h) for t, h in outs if any(t is u for u in [d["loss"]] + d["grads"])] for d in st]

    def copy_in(p, after_event):
        """Copy one step's inputs into buffer set p (after `after_event`); per-linear events."""
        if after_event is not None:
            copier.wait_event(after_event)
        xd, ytd = sets[p]
        ready, seen = [], set()
        with torch.cuda.stream(copier):
            for i in range(len(st)):
                if keys[i] not in seen:
                    seen.add(keys[i])
                    xd[keys[i]].copy_(xs_h[keys[i]], non_blocking=True)
                ytd[i].copy_(yts_h[i], non_blocking=True)
                e = torch.cuda.Event()
                e.record(copier)
                ready.append(e)
        return ready

    def run(nsteps):
        """nsteps steps; step 0's copies first, then each step's copies during the previous."""
        ready = copy_in(0, None)
        done_prev = None
        for t in range(nsteps):
            p = t % 2
            xd, ytd = sets[p]
            for i, d in enumerate(st):
                d["X"], d["Yt"] = xd[keys[i]], ytd[i]
            nxt = copy_in(1 - p, done_prev) if t + 1 < nsteps else None

            def before(i, ready=ready):
                torch.cuda.current_stream().wait_event(ready[i])

            def after(i):
                for tt, h in out_of[i]:
                    h.copy_(tt, non_blocking=True)

            step(before=before, after=after)
            done_prev = torch.cuda.Event()
            done_prev.record(main)
            ready = nxt
        for i, d in enumerate(st):  # leave the bench's own tensors in place
            d["X"], d["Yt"] = sets[0][0][keys[i]], sets[0][1][i]

    steps = max(3, args.steps // 2)
    run(2)
    barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    run(steps)
    b.record()
    barrier()
    ms = max_over_ranks(a.elapsed_time(b) / steps, world, dev)
    return {"value": job_throughput(flops_step, ms, world), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "steps": steps,
            "pipeline": "inputs double-buffered: step t + 1's copies overlap step t's kernels"}


def run_only(args):
    """One secondary measurement alone on GPU 0 (used by the ncu commands under profiles/)."""
    import torch

    from paper_2606_26650_gb300 import catq as C
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks = measured_peaks()
    wl = syn.WORKLOADS[DEFAULT_WORKLOAD]

    def barrier():
        torch.cuda.synchronize()

    if args.only == "moe":
        r = measure_moe(C, torch, dev, peaks, 1, args.s, steps=args.steps, warmup=args.warmup,
                        experts=args.moe_experts, nstreams=args.streams)
    elif args.only.startswith("decode_b"):
        rows = int(args.only[len("decode_b"):].split("_")[0])
        r = measure_decode(C, torch, wl, dev, peaks, rows=rows, steps=args.steps, staged="staged" in args.only)
    else:
        bw = syn.WORKLOADS[args.workload] if args.workload in BLOCK_WINDOW_SHAPES else wl
        r = measure_block_window(C, torch, bw, dev, peaks, 1, args.s, barrier, steps=args.steps, warmup=args.warmup,
                                 streams=args.streams)
    print(json.dumps({"only": args.only, **r}), flush=True)


def main():
    args = parse()
    if args.only:
        run_only(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
