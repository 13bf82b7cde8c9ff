"""The benchmark's multi-rank plumbing (max elapsed over ranks, units summed
over ranks, barrier-bracketed timed region) on CPU ranks with gloo, and the
reference arm (the CPU oracle) end to end.  No GPU is used here."""
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


def _rank_main(rank, world, port, q):
    import time

    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)

    def barrier():
        dist.barrier()

    def rmax(x):
        t = torch.tensor([float(x)])
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    def rsum(x):
        t = torch.tensor([float(x)], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.SUM)
        return int(t.item())

    calls = []
    # rank 1 is slower per step: the combined time must be rank 1's
    step = lambda: (calls.append(1), time.sleep(0.01 * (1 + rank)))
    elapsed = bench.run_timed(step, steps=5, warmup=3, sync=lambda: None, barrier=barrier)
    t, units = bench.combine_ranks(elapsed, 1000 * (rank + 1), world, rmax, rsum)
    q.put((rank, elapsed, t, units, len(calls)))
    dist.destroy_process_group()


def test_two_gloo_ranks_combine():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, e0, t0, u0, c0), (r1, e1, t1, u1, c1) = res
    assert c0 == c1 == 8                              # 3 warm-up + 5 timed steps on each rank
    assert t0 == t1 == pytest.approx(max(e0, e1))     # max over ranks, same on every rank
    assert min(e0, e1) >= 5 * 0.02 * 0.95             # the closing barrier holds rank 0 until rank 1 is done
    assert u0 == u1 == 3000                           # units of both ranks


def test_reference_arm_runs_on_cpu():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "3", "--kernels", "20000"], capture_output=True, text=True, env=env,
                         timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "M kernels/s" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == (os.cpu_count() or 1)
    assert line["config"]["kernels"] == 20000 and line["config"]["same_config"] is False
    assert line["e2e"]["h2d_bytes_per_step"] == 0
