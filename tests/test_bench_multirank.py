"""The bench's multi-rank host logic on CPU: two gloo ranks, no GPU.

Every rank runs its own batch (weak scaling, no data exchange); the step time is
the maximum over ranks and the reported value is the whole job's bytes over that
time.  The reference arm prints from rank 0 only.
"""
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r measured (r + 1) * 10 ms for 100 steps: the job's step time is the slowest rank's
        total = bench.max_over_ranks(10.0 * (rank + 1), world, "cpu")
        launch = bench.max_over_ranks(0.05 * (rank + 1), world, "cpu")
        r = {"w": bench.WORKLOAD, "total_ms": total, "launch_ms": launch, "fp32_launch_ms": 0.2, "e2e_ms": 0.3,
             "h2d": 1, "d2h": 1, "clocks": None, "bits": 9.5, "dev_name": "cpu"}
        line = bench.make_line(r, 100, 5, world)
        out[rank] = (total, line["value"], line["n_gpus"], line["scaling"])
    finally:
        dist.destroy_process_group()


def test_two_rank_max_and_weak_scaling_value():
    port = _free_port()
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    import bench
    bytes_step = bench.algorithmic_bytes(bench.WORKLOAD)
    for rank in range(2):
        total, value, n, scaling = out[rank]
        assert total == 20.0
        assert n == 2 and scaling == "weak"
        assert value == pytest.approx(2 * bytes_step / (20.0 / 100 * 1e-3) / 1e12)


def test_reference_arm_prints_from_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "3"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_bench_line_carries_the_contract_keys():
    """The JSON line of one rank: every key the bench contract names, with its type."""
    sys.path.insert(0, ROOT)
    import json

    import bench
    r = {"w": bench.WORKLOAD, "total_ms": 8.0, "launch_ms": 0.08, "fp32_launch_ms": 0.2, "e2e_ms": 0.085,
         "h2d": 10, "d2h": 4, "clocks": {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}, "bits": 9.5,
         "dev_name": "cpu", "reps_ms": [0.08] * 5, "graph_ms": 0.079}
    line = json.loads(json.dumps(bench.make_line(r, 100, 5, 1)))
    for key, typ in (("metric", str), ("value", float), ("unit", str), ("n_gpus", int), ("steps", int),
                     ("warmup", int), ("ms_per_step", float), ("higher_is_better", bool), ("scaling", str),
                     ("dtype", str), ("data", str), ("config", dict), ("clocks", dict), ("e2e", dict),
                     ("gpu_launches", int), ("roofline", dict)):
        assert isinstance(line[key], typ), key
    assert "vs_baseline" in line and line["config"]["workload"] == bench.WORKLOAD.name
    assert set(line["e2e"]) >= {"value", "unit", "h2d_bytes_per_step", "d2h_bytes_per_step"}
    assert set(line["roofline"]) >= {"bound", "achieved", "peak", "unit", "frac", "traffic"}
    assert line["roofline"]["frac"] == pytest.approx(line["roofline"]["achieved"] / line["roofline"]["peak"])
    assert line["value"] == pytest.approx(bench.algorithmic_bytes(bench.WORKLOAD) / 0.08e-3 / 1e12)
