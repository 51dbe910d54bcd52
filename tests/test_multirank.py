"""The N > 1 path of bench.py on CPU: two gloo ranks reduce their timings
to the slowest rank's, the whole-job throughput counts every rank's bytes
(weak scaling), every rank draws its own replica, and under torchrun the
reference arm runs on rank 0 alone and prints one line."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from paper_2606_00724_gb300 import synth  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    torch.distributed.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                                         world_size=world)
    try:
        got = bench.max_over_ranks([1.0 + rank, 10.0 - rank, 3.5], "cpu")
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump(got, f)
    finally:
        torch.distributed.destroy_process_group()


def test_max_over_ranks_gloo(tmp_path):
    port = _free_port()
    mp.start_processes(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    for rank in range(2):
        assert json.load(open(tmp_path / f"rank{rank}.json")) == [2.0, 10.0, 3.5]


def test_max_over_ranks_single_process():
    assert bench.max_over_ranks([4.0, 5.0], "cpu") == [4.0, 5.0]


def test_weak_scaling_aggregate():
    ms1, v1 = bench.aggregate(1, 2e8, 100.0, 10)
    ms2, v2 = bench.aggregate(2, 2e8, 100.0, 10)
    assert ms1 == ms2 == 10.0
    assert v1 == pytest.approx(20.0) and v2 == pytest.approx(2 * v1)


def test_ranks_draw_different_replicas():
    w = synth.WORKLOADS["c1"]
    a = bench.make_inputs(w, "c1", "cpu", 0)[0]
    b = bench.make_inputs(w, "c1", "cpu", 1)[0]
    a2 = bench.make_inputs(w, "c1", "cpu", 0)[0]
    assert torch.equal(a.K, a2.K) and not torch.equal(a.K, b.K)


def test_reference_arm_under_torchrun():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"), "--impl", "reference",
           "--workload", "c1", "--steps", "1", "--warmup", "3", "--gpus", "2"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, res.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
