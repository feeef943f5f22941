"""The N > 1 bench path on the CPU: world-size-2 `gloo` ranks (no GPU).

`bench.py --gpus N` under torchrun runs N independent replicas; the only
cross-rank steps are a barrier and the max of the ranks' timed totals, from
which the whole-job value is computed.  Here two spawned ranks run the same
aggregation over gloo with different local times, and the reference arm's
non-zero ranks are checked to exit without work.
"""
from __future__ import annotations

import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, ws, port, local_ms, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    sys.path.insert(0, ROOT)
    import bench

    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        dist.barrier()
        total, e2e, value, e2e_value = bench.aggregate_ranks(local_ms[rank], 2 * local_ms[rank], ws, 1024, 10,
                                                             torch.device("cpu"))
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{total!r} {e2e!r} {value!r} {e2e_value!r}\n")
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("local_ms", [(10.0, 12.5), (7.0, 3.0)])
def test_two_ranks_take_the_slowest_rank(tmp_path, local_ms):
    ws = 2
    mp.start_processes(_rank_main, args=(ws, _free_port(), local_ms, str(tmp_path)), nprocs=ws, join=True,
                       start_method="spawn")
    slowest = max(local_ms)
    for rank in range(ws):
        total, e2e, value, e2e_value = map(float, open(tmp_path / f"rank{rank}.txt").read().split())
        assert total == slowest and e2e == 2 * slowest  # every rank reports the max
        # weak scaling: both ranks' 10 steps x 1,024 tokens over the slowest rank's time
        assert value == pytest.approx(ws * 1024 * 10 / (slowest / 1e3), rel=1e-12)
        assert e2e_value == pytest.approx(ws * 1024 * 10 / (2 * slowest / 1e3), rel=1e-12)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    total, e2e, value, _ = bench.aggregate_ranks(4.0, 8.0, 1, 1024, 2, torch.device("cpu"))
    assert (total, e2e) == (4.0, 8.0) and value == pytest.approx(1024 * 2 / 4e-3)


def test_reference_arm_other_ranks_exit_without_work():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2"],
                       capture_output=True, text=True, env=env, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""


def test_replica_plan():
    """The bench's replica plan: the single image gets one table replica per
    stream (sixteen), the batched table two, and tables that cannot be held
    several times (or are not HBM-resident) one with L2 flushed."""
    import bench
    from paper_2607_16305_gb300 import workloads as W

    assert bench.plan_replicas(W.WORKLOADS["single_image"]) == (16, 16)
    assert bench.plan_replicas(W.WORKLOADS["batched_zipf"]) == (2, 2)
    assert bench.plan_replicas(W.WORKLOADS["large_table"]) == (1, 1)
    assert bench.plan_replicas(W.WORKLOADS["multilayer_host"]) == (1, 1)
    for w in W.WORKLOADS.values():
        r, ns = bench.plan_replicas(w)
        assert r % ns == 0 and r * bench.table_bytes(w) <= max(bench.REPLICA_BUDGET, bench.table_bytes(w))
