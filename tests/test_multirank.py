"""The multi-rank host logic of bench.py on CPU: two gloo ranks, as torchrun would launch
them (one replica of the step per rank; no collective on the data path).  Checks the
max-over-ranks timing, the barrier, the whole-job throughput and that only rank 0 of the
reference arm prints."""

import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, _ = bench.dist_env()
    bench.barrier(w)
    ms = bench.max_over_ranks(10.0 + 5.0 * r, w)                 # rank 1 is the slow one
    value = bench.job_throughput(1e9, 100, w, ms)
    dist.destroy_process_group()
    q.put((r, w, ms, value))


def test_two_gloo_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(2))
    for r, w, ms, value in res:
        assert w == 2 and ms == 15.0                               # max over ranks, on every rank
        assert value == pytest.approx(2 * 1e9 * 100 / 0.015 / 1e9)   # both replicas' bytes / slowest time


def test_reference_arm_prints_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", OMP_NUM_THREADS="1")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                          "--config", "tiny_1k", "--steps", "1", "--warmup", "3"], env=env, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0 and out.stdout.strip() == ""
    env.update(RANK="0", LOCAL_RANK="0")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                          "--config", "tiny_1k", "--steps", "1", "--warmup", "3"], env=env, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    # the reference line's contract: the oracle as cpu_baseline, an e2e without copies
    assert line["unit"] == "GB/s" and line["higher_is_better"] is True and line["steps"] == 1
    assert line["config"]["workload"] == "tiny_1k"
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == line["value"]
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["unit"] == line["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0
