"""The N>1 bench path on CPU: two gloo ranks and a torchrun launch of the reference arm.

The decode step shards by sequence: every rank decodes its own batch and no
data crosses ranks; the only collective is the max over ranks of the timed
region, which these tests run over gloo with world size 2.
"""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # rank r was slower on the first timer and faster on the second
        got = bench.max_over_ranks([10.0 + rank, 7.0 - 3.0 * rank])
        value = bench.job_tokens_per_s(world, 16, 5, got[0])
        with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
            json.dump({"max": got, "value": value}, f)
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo(tmp_path):
    port = _free_port()
    mp.start_processes(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    res = [json.load(open(tmp_path / f"r{r}.json")) for r in range(2)]
    for r in res:
        assert r["max"] == [11.0, 7.0]
        # 2 ranks x 16 sequences x 5 steps over the slowest rank's 11 ms
        assert r["value"] == pytest.approx(2 * 16 * 5 / 11e-3)


def test_max_over_ranks_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks([3.0, 4.5]) == [3.0, 4.5]
    assert bench.job_tokens_per_s(1, 8, 10, 20.0) == pytest.approx(4000.0)


def test_reference_arm_under_torchrun():
    """torchrun with 2 ranks: rank 0 alone runs the oracle and prints one line; rank 1 exits 0."""
    port = _free_port()
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="", OMP_NUM_THREADS="2")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--config", "c1", "--gpus", "2", "--steps", "2", "--warmup", "3"]
    r = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["steps"] == 2 and d["warmup"] == 3
    # the workload is named as in the timed arm's line
    assert d["config"]["name"] == "c1" and d["config"]["workload"] != "c1"
    assert d["value"] > 0 and d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
