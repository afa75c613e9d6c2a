"""The multi-process host logic of bench.py on CPU: world_size-2 gloo ranks
(the timing reduction, the barrier, per-rank replica inputs) and the
reference arm launched the way the benchmark driver launches it (torchrun,
rank 0 alone prints one JSON line, the other ranks exit 0 without work)."""
import json
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


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    from paper_2108_00951_gb300 import workloads
    dist = bench.dist_init("gloo")
    assert dist is not None and bench.dist_env() == (rank, world, rank)
    # rank r spent 1 + 1.5 r seconds on 10 + 22 r units
    seconds, units = bench.reduce_timing(dist, 1.0 + 1.5 * rank, 10.0 + 22.0 * rank)
    bench.barrier(dist)
    w = bench.replica_workload(workloads.BY_NAME["lr"], rank)
    g = workloads.gradient(w, 0, 0)
    seeds = [None] * world
    dist.all_gather_object(seeds, (w.seed, float(g[:64].sum())))
    with open(os.path.join(out_dir, "rank%d.json" % rank), "w") as f:
        json.dump({"seconds": seconds, "units": units, "seeds": seeds}, f)
    dist.destroy_process_group()


def test_two_gloo_ranks_reduce_timing_and_replicas(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    res = [json.load(open(tmp_path / ("rank%d.json" % r))) for r in range(world)]
    for r in res:
        assert r["seconds"] == pytest.approx(2.5)      # max over ranks
        assert r["units"] == pytest.approx(42.0)       # sum over ranks
    seeds = res[0]["seeds"]
    assert seeds == res[1]["seeds"]
    assert seeds[0][0] != seeds[1][0]                  # each rank draws its own inputs
    assert seeds[0][1] != seeds[1][1]


def test_single_rank_needs_no_process_group(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    for v in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(v, raising=False)
    assert bench.dist_env() == (0, 1, 0)
    assert bench.dist_init("gloo") is None
    assert bench.reduce_timing(None, 3.0, 7.0) == (3.0, 7.0)
    bench.barrier(None)


def test_reference_arm_under_torchrun_prints_one_line_from_rank_0():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "lr",
           "--gpus", "2", "--steps", "3", "--warmup", "1"]
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1, p.stdout
    out = json.loads(lines[0])
    assert out["impl"] == "reference" and out["unit"] == "GB/s" and out["value"] > 0
    assert out["n_gpus"] == 2 and out["steps"] == 3 and out["warmup"] == 1
    assert out["cpu_baseline"]["kind"] == "oracle" and out["cpu_baseline"]["value"] == out["value"]
    assert out["e2e"] == {"value": out["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                          "d2h_bytes_per_step": 0}
