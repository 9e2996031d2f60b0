"""bench.py's host logic on the CPU: the multi-rank path (two `gloo` ranks) and the
sequencing of the factor update that closes each step.

Each rank runs the same step on its own seeded inputs (independent replicas, weak scaling),
the step time is the slowest rank's, and the job's throughput is the ranks' total work over
that time.  The CUDA kernels take no part in this; the GPU runs use the same functions with
the NCCL backend.
"""
import json
import os
import socket

import numpy as np
import pytest

import bench
from paper_2606_26650_gb300 import synthetic as syn

torch = pytest.importorskip("torch")

WORLD = 2
STEP_MS = {0: 10.0, 1: 15.0}  # the second rank is the slow one
FLOPS = 1.0e12


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, port: int, out_dir: str) -> None:
    import torch.distributed as dist

    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(WORLD),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=WORLD)
    try:
        r, local, world = bench.dist_env()
        ms = bench.max_over_ranks(STEP_MS[r], world, torch.device("cpu"))
        value = bench.job_throughput(FLOPS, ms, world)
        wl = syn.WORKLOADS["c3_llama3_8b_block"]
        x = syn.activations(wl, "x_hidden", 4, 64, seed=r)
        shards = [None] * world
        dist.all_gather_object(shards, x.tolist())
        dist.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"rank": r, "local": local, "world": world, "ms": ms, "value": value,
                       "shards": shards}, f)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp

    port = _free_port()
    mp.start_processes(_rank_main, args=(port, str(tmp_path)), nprocs=WORLD, join=True, start_method="spawn")
    res = [json.loads((tmp_path / f"rank{r}.json").read_text()) for r in range(WORLD)]
    for r, d in enumerate(res):
        assert (d["rank"], d["local"], d["world"]) == (r, r, WORLD)
        # every rank reports the slowest rank's time and the whole job's throughput
        assert d["ms"] == max(STEP_MS.values())
        assert d["value"] == pytest.approx(WORLD * FLOPS / (15.0e-3) / 1e12)
    # ranks work on different, reproducible inputs (seeded by rank)
    a, b = (np.asarray(s) for s in res[0]["shards"])
    assert not np.array_equal(a, b)
    wl = syn.WORKLOADS["c3_llama3_8b_block"]
    np.testing.assert_array_equal(a, syn.activations(wl, "x_hidden", 4, 64, seed=0))
    np.testing.assert_array_equal(b, syn.activations(wl, "x_hidden", 4, 64, seed=1))


def test_single_rank_is_unchanged():
    assert bench.max_over_ranks(12.5, 1, None) == 12.5
    assert bench.job_throughput(2.0e12, 4.0, 1) == pytest.approx(500.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = bench.parse(["--impl", "reference", "--steps", "1", "--warmup", "0"])
    assert bench.run_reference(args) is None
    assert capsys.readouterr().out == ""


def test_factor_update_sequence_of_the_bench_step():
    """bench.py's step closes with one AdamW update per linear: the update count rises by
    one per step, the learning rate follows the linear decay of App. B.1 through the
    library's host call, a full calibration's updates later a fresh calibration starts (count
    1, zero moments), and every linear gets its own moments of 6 G floats."""
    from paper_2606_26650_gb300 import catq as C

    calls = []

    class FakeC:
        adamw = staticmethod(C.adamw)
        catq_linear_decay_lr = staticmethod(C.catq_linear_decay_lr)

        @staticmethod
        def catq_factor_adamw_step(*args):
            calls.append(args)

    class L:
        d_mu, d_alpha, d_delta = "mu", "alpha", "delta"

    upd = bench.FactorUpdate(FakeC, torch, torch.device("cpu"), [4, 6])
    assert [m.numel() for m in upd.moments] == [24, 36]
    lrs = []
    for _ in range(3):
        upd.advance()
        lrs.append(upd.lr)
        upd.apply(1, L, ["g0", "g1", "g2"])
    assert lrs[0] == pytest.approx(bench.LR0)
    assert lrs[1] == pytest.approx(bench.LR0 * (1 - 1 / bench.UPDATES), rel=1e-6)
    assert [c[-2] for c in calls] == [1, 2, 3]                   # update count t
    assert calls[0][:6] == ("mu", "alpha", "delta", "g0", "g1", "g2")
    assert calls[0][6] is upd.moments[1]
    upd.moments[1].fill_(0.5)
    upd.t = bench.UPDATES
    upd.advance()
    assert upd.lr == pytest.approx(bench.LR0)                     # a fresh calibration starts:
    assert upd.t == 1                                             # first update again (bias correction)
    assert not upd.moments[1].any()                               # and zero moments
