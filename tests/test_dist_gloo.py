"""The multi-rank host logic of bench.py on two gloo ranks (CPU): scene
shards are disjoint and cover the job, the job's time is the slowest rank's,
the aggregate throughput counts every rank's bytes, and the reference arm runs
on rank 0 only. The data path itself has no collective (scenes are
independent), so nothing else crosses ranks."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        scenes = bench.scenes_of_rank(2, rank)
        gathered = [None] * world
        dist.all_gather_object(gathered, scenes)
        local_ms = [1.25, 3.5][rank]
        job_ms = bench.max_over_ranks(local_ms, world)
        value = bench.aggregate_gbs(1e9, world, job_ms)
        with open(os.path.join(out_dir, "rank%d.json" % rank), "w") as f:
            json.dump({"scenes": gathered, "job_ms": job_ms, "value": value}, f)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    res = [json.load(open(tmp_path / ("rank%d.json" % r))) for r in range(world)]
    for r in res:
        flat = [s for part in r["scenes"] for s in part]
        assert sorted(flat) == list(range(4)) and len(set(flat)) == 4  # disjoint, covering
        assert r["job_ms"] == 3.5                                         # the slowest rank
        assert abs(r["value"] - 2 * 1e9 / 3.5e-3 / 1e9) < 1e-9            # all ranks' bytes
    assert res[0]["scenes"][0] != res[0]["scenes"][1]  # each rank its own scenes


def test_scenes_differ_between_ranks():
    # rank r verifies scene r: different clips, not the same data replicated
    sys.path.insert(0, ROOT)
    import numpy as np
    from paper_2606_31160_gb300 import workloads
    a = workloads.target_layer(layer=0, ell=[3], scene=0)
    b = workloads.target_layer(layer=0, ell=[3], scene=1)
    assert not np.array_equal(a.q.float().numpy(), b.q.float().numpy())
    c = workloads.target_layer(layer=0, ell=[3])
    assert np.array_equal(a.q.float().numpy(), c.q.float().numpy())  # scene 0 is the default


@pytest.mark.parametrize("rank", [0, 1])
def test_reference_arm_prints_on_rank_zero_only(rank):
    env = dict(os.environ, WORLD_SIZE="2", RANK=str(rank), LOCAL_RANK=str(rank))
    res = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "3",
                          "--gpus", "2"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    if rank == 0:
        assert len(lines) == 1
        line = json.loads(lines[0])
        assert line["impl"] == "reference" and line["n_gpus"] == 2
        # the line a bench arm prints: same metric and unit as ours, the oracle
        # described as the cpu baseline, an e2e object with no host copies
        for key in ("metric", "value", "unit", "steps", "warmup", "ms_per_step", "higher_is_better",
                    "scaling", "dtype", "data", "config", "cpu_baseline", "e2e"):
            assert key in line, key
        assert line["unit"] == "GB/s" and line["higher_is_better"] is True and line["warmup"] >= 3
        assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
        assert line["cpu_baseline"]["value"] == line["value"] and line["cpu_baseline"]["sample"]
        assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
        assert line["e2e"]["value"] == line["value"] and line["e2e"]["unit"] == line["unit"]
    else:
        assert lines == []
