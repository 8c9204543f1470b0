"""N > 1 host logic of bench.py on CPU: two gloo ranks, no GPU.

Each rank is an independent replica (the compare shards with no data-path
collective); the only exchange is the max over ranks of the timed interval,
and the whole-job value counts the pairs of every rank.
"""
import json
import os
import socket
import subprocess
import sys
from pathlib import Path

ROOT = Path(__file__).resolve().parent.parent

CHILD = r"""
import json, os, sys
sys.path.insert(0, sys.argv[1])
import torch.distributed as dist
import bench
rank, world, local = bench.dist_env()
dist.init_process_group("gloo")
dist.barrier()
ms = bench.max_over_ranks(10.0 + 5.0 * rank, "cpu")
value = bench.whole_job_rate(1000, world, 4, ms)
print(json.dumps({"rank": rank, "world": world, "local": local, "ms": ms, "value": value}))
dist.destroy_process_group()
"""


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_take_max_time_and_count_every_rank():
    port = free_port()
    procs = []
    for r in range(2):
        env = dict(os.environ, RANK=str(r), LOCAL_RANK=str(r), WORLD_SIZE="2", MASTER_ADDR="127.0.0.1",
                   MASTER_PORT=str(port))
        procs.append(subprocess.Popen([sys.executable, "-c", CHILD, str(ROOT)], env=env, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=240)
        assert p.returncode == 0, err
        outs.append(json.loads(out.strip().splitlines()[-1]))
    for o in outs:
        assert o["world"] == 2
        assert o["ms"] == 15.0  # the slower replica's time, on every rank
        assert abs(o["value"] - 1000 * 2 * 4 / 15e-3) < 1e-6
    assert sorted(o["rank"] for o in outs) == [0, 1]


def test_single_process_is_identity():
    sys.path.insert(0, str(ROOT))
    import bench
    assert bench.max_over_ranks(3.5, "cpu") == 3.5
    assert bench.whole_job_rate(10, 1, 2, 1000.0) == 20.0
