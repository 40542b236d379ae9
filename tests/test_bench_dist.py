"""The multi-rank logic of bench.py on CPU: two gloo ranks (127.0.0.1)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = 10.0 + 5.0 * rank                       # rank 1 is the slow one
    slow = bench.slowest_ms(ms, world, "cpu")
    val = bench.job_throughput(1000, world, slow)
    q.put((rank, slow, val, bench.rank_seed_offset(rank)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_take_the_slowest_and_sum_the_batches():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, slow, val, seed in out:
        assert slow == 15.0                       # max over ranks
        assert val == pytest.approx(2 * 1000 / 0.015)   # both ranks' tokens, slowest time
    assert [o[3] for o in out] == [0, 1]          # distinct batches per rank


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.slowest_ms(12.5, 1, "cpu") == 12.5
    assert bench.job_throughput(500, 1, 2.0) == pytest.approx(250000.0)


def _run_bench(args, env_extra=None):
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ)
    env.update(env_extra or {})
    res = subprocess.run([sys.executable, os.path.join(root, "bench.py"), *args], capture_output=True,
                         text=True, env=env, timeout=600, cwd=root)
    return res


def test_reference_arm_prints_the_oracle_line():
    """`bench.py --impl reference` times the CPU oracle on all host cores and prints one JSON line
    with the bench's metric, unit and config, a cpu_baseline describing the run, and an e2e
    block with no host-device traffic."""
    import json
    res = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "3", "--workload", "tiny_kda"])
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.strip()]
    assert len(lines) == 1, res.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] == 3
    assert d["config"]["workload"] == "tiny_kda"
    cb = d["cpu_baseline"]
    import os
    cores = len(os.sched_getaffinity(0))   # the oracle's timing build runs on every usable core
    assert cb["kind"] == "oracle" and cb["cores"] == cores and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_print_nothing():
    res = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "3", "--workload", "tiny_kda"],
                     {"RANK": "1", "WORLD_SIZE": "2"})
    assert res.returncode == 0, res.stderr[-2000:]
    assert res.stdout.strip() == ""
