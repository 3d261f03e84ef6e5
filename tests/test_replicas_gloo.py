"""The N > 1 path of the benchmark on CPU: world_size-2 `gloo` process groups.

The layer step has no exchange, so N GPUs run N independent replicas.  What the
ranks share is only the bookkeeping: a barrier on both sides of the timed
region, the maximum of the per-rank totals, and the whole-job value computed
from that maximum.  These tests run that bookkeeping (the helpers bench.py
uses) on two gloo ranks, and check that two replicas of the (oracle) step on
the same seeded inputs produce identical bytes.
"""
import hashlib
import os
import socket
import sys
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")
dist = pytest.importorskip("torch.distributed")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from oracle import method as om
        from paper_2408_14267_gb300 import workloads as wl

        # timed region as bench.py brackets it; rank 1 is made the slow one
        steps, ops = 4, 1.0e9
        dist.barrier()
        t0 = time.perf_counter()
        local = []
        for _ in range(steps):
            s0 = time.perf_counter()
            time.sleep(0.01 * (rank + 1))
            local.append((time.perf_counter() - s0) * 1e3)
        dist.barrier()
        wall_ms = (time.perf_counter() - t0) * 1e3
        total = bench.max_over_ranks(sum(local))
        value = bench.job_tops(ops, steps, world, total)

        # one replica of the layer step on every rank, same seeded inputs
        w = wl.linear_small()
        out = om.layer_step_linear(w["x"], w["w"], w["gamma"], w["gy"], w["bits_s"], w["mode_s"], w["seed_s"],
                                   w["bits_c"], w["mode_c"], w["seed_c"], rows_per_group=w["rows_per_group"])
        h = hashlib.sha256()
        for k in ("y", "dx", "dw"):
            h.update(np.ascontiguousarray(out[k]).tobytes())
        digests = [None] * world
        dist.all_gather_object(digests, h.hexdigest())
        np.save(os.path.join(out_dir, f"rank{rank}.npy"),
                np.array([sum(local), total, value, wall_ms], dtype=np.float64))
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write("\n".join(digests))
    finally:
        dist.destroy_process_group()


def test_two_replicas_max_over_ranks_and_job_value(tmp_path):
    world = 2
    torch.multiprocessing.spawn(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    r = [np.load(tmp_path / f"rank{i}.npy") for i in range(world)]
    local = [x[0] for x in r]
    # every rank holds the slowest rank's total
    for x in r:
        assert x[1] == max(local)
    assert local[1] > local[0]
    # whole-job value: all ranks' work over the slowest rank's time
    import bench
    expect = bench.job_tops(1.0e9, 4, world, max(local))
    for x in r:
        assert x[2] == pytest.approx(expect, rel=1e-12)
    # both replicas of the step are identical, byte for byte
    d = [open(tmp_path / f"rank{i}.txt").read().split() for i in range(world)]
    assert d[0] == d[1] and d[0][0] == d[0][1]


def test_single_process_helpers_need_no_process_group():
    import bench
    assert not dist.is_initialized()
    assert bench.max_over_ranks(3.5) == 3.5
    # 6 M K D operations per step at 0.1 ms per step: 1 GPU and 8 replicas
    ops = 6.0 * 8192 * 2304 * 256
    assert bench.job_tops(ops, 10, 1, 1.0) == pytest.approx(ops * 10 / 1e-3 / 1e12)
    assert bench.job_tops(ops, 10, 8, 1.0) == pytest.approx(8 * ops * 10 / 1e-3 / 1e12)


def test_reference_arm_other_ranks_do_no_work(capsys):
    """Under torchrun only rank 0 runs the oracle and prints; other ranks exit without work."""
    import argparse

    import bench
    args = argparse.Namespace(steps=1, warmup=0, impl="reference", gpus=2)
    t0 = time.perf_counter()
    assert bench.reference_arm(args, world=2, rank=1) is None
    assert time.perf_counter() - t0 < 1.0
    assert capsys.readouterr().out == ""
