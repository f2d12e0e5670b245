"""The N > 1 host path of bench.py on CPU: two gloo ranks on 127.0.0.1 (one process per rank, as
torchrun launches the GPU arm). Timing is aggregated as the maximum over ranks, all ranks pass the
barrier, every rank gets its own input batch (weak scaling, no collective on the data path), the
whole-job value counts every rank's work over the slowest rank's time; and the reference arm under
two ranks prints exactly one line (rank 0) while rank 1 exits cleanly."""
import json
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


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        sys.path.insert(0, ROOT)
        import bench
        local_ms = 100.0 + 50.0 * rank          # rank 1 is the slower one
        m = bench.max_over_ranks(local_ms, world)
        bench.barrier(world)
        out[rank] = (m, bench.rank_input_seed(rank))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_aggregate_max_time_and_distinct_batches():
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    assert out[0][0] == out[1][0] == 150.0            # both ranks see the slowest rank's time
    assert out[0][1] != out[1][1]                      # each rank runs its own batch
    sys.path.insert(0, ROOT)
    import bench
    # whole-job value: 2 ranks x 3 steps x 1e12 FLOPs in 150 ms
    assert bench.weak_scaling_value(1e12, 3, 2, 150.0) == pytest.approx(2 * 3 / 0.150)
    assert bench.max_over_ranks(7.0, 1) == 7.0         # N = 1: no collective at all


def test_reference_arm_under_two_ranks_prints_once():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes", "1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
