"""CPU checks of the benchmark's host logic: the reference arm (the CPU oracle
on a bounded sample) prints one well-formed JSON line, and the multi-rank
timing aggregation (max of times, sum of work) is right on 2 gloo ranks."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("workload,prefix", [(None, "leduc_holdem_64x64"),
                                              ("kuhn", "kuhn_4x4"),
                                              ("spread3", "spread_n3_4096env")])
def test_reference_arm_json_line(workload, prefix):
    """The reference arm times the oracle on the GPU arm's own workload (the
    default is the 64 x 64 bf16 Leduc sweep) and prints one JSON line."""
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
           "--steps", "2", "--warmup", "1"]
    if workload:
        cmd += ["--workload", workload]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
    assert d["config"]["workload"].startswith(prefix)


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    mx = bench.max_over_ranks(10.0 + rank, world)
    sm = bench.sum_over_ranks(100.0 * (rank + 1), world)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, mx, sm))


def test_rank_aggregation_gloo():
    import multiprocessing as mp
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(120)
    assert all(p.exitcode == 0 for p in ps)
    out = sorted(q.get() for _ in range(2))
    assert out == [(0, 11.0, 300.0), (1, 11.0, 300.0)]
