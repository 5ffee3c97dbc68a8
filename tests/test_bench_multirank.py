"""bench.py's multi-rank host logic on CPU: two gloo ranks.

Pairs are independent, so the ranks shard the batches with no data-path
collective; the only exchanges are the timing barrier and two scalar
reductions (max of the elapsed time, sum of the pairs scored).  These tests
run that logic as two processes on the gloo backend, and the reference arm
under a two-rank launch, where rank 0 alone prints its line.
"""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    n_batches, steps = 10, 5
    mine = [bench.shard_batch(rank, world, s, n_batches) for s in range(steps)]
    # rank r scored 100 * (r + 1) pairs in 10 * (r + 1) ms
    t_max = bench.reduce_over_ranks(dist, 10.0 * (rank + 1), "max", "cpu")
    pairs = bench.reduce_over_ranks(dist, 100.0 * (rank + 1), "sum", "cpu")
    dist.barrier()
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"mine": mine, "t_max": t_max, "pairs": pairs}, f)
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_batches_and_reduce(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    # every step: the ranks take different batches, and over the steps no batch repeats
    for s in range(5):
        assert res[0]["mine"][s] != res[1]["mine"][s]
    flat = res[0]["mine"] + res[1]["mine"]
    assert sorted(flat) == list(range(10))
    for r in res:
        assert r["t_max"] == 20.0  # slowest rank's time
        assert r["pairs"] == 300.0  # all ranks' pairs
    # whole-job throughput = all pairs / slowest rank's time
    assert res[0]["pairs"] / (res[0]["t_max"] / 1e3) == pytest.approx(15000.0)


def test_world_size_one_reduction_is_identity():
    assert bench.reduce_over_ranks(None, 3.5, "max", "cpu") == 3.5
    assert bench.reduce_over_ranks(None, 3.5, "sum", "cpu") == 3.5
    assert [bench.shard_batch(0, 1, s, 4) for s in range(6)] == [0, 1, 2, 3, 0, 1]


def test_reference_arm_under_two_ranks_prints_one_line():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py", "--impl", "reference",
           "--workload", "qwen3-0.6b-2l", "--steps", "2", "--warmup", "1", "--cpu-seconds", "2"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600,
                       env=dict(os.environ, CUDA_VISIBLE_DEVICES=""))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0


def test_config_numbers_select_the_workloads():
    from paper_2609_03311_gb300 import synth

    assert set(bench.CONFIG_WORKLOADS.values()) == set(synth.WORKLOADS)
    assert bench.parse_args(["--config", "3'"]).workload == "qwen3-8b-m64"
    assert bench.parse_args(["--config", "2"]).workload == "qwen3-4b"
    assert bench.parse_args([]).workload == "qwen3-8b-m64"  # the headline by default
