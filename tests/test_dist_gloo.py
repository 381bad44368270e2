"""The benchmark's multi-rank host logic on CPU (gloo, world size 2): ranks
run independent replicas, the timed duration is the max over ranks, and the
reference arm runs on rank 0 only."""
import json
import os
import socket
import subprocess
import sys

import pytest

from conftest import ROOT


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


WORKER = r"""
import os, sys, json
sys.path.insert(0, ROOT)
import bench
d = bench.Dist()
v = d.max(1.0 + d.rank)          # rank r reports 1 + r seconds
d.barrier()
print(json.dumps({"rank": d.rank, "world": d.world, "max": v}))
d.close()
"""


def test_max_over_ranks_gloo():
    port = _free_port()
    procs = []
    for r in range(2):
        env = dict(os.environ, RANK=str(r), LOCAL_RANK=str(r), WORLD_SIZE="2",
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), CUDA_VISIBLE_DEVICES="")
        procs.append(subprocess.Popen([sys.executable, "-c", WORKER.replace("ROOT", repr(ROOT))],
                                      env=env, stdout=subprocess.PIPE, stderr=subprocess.PIPE,
                                      text=True))
    outs = [p.communicate(timeout=120) for p in procs]
    for p, (o, e) in zip(procs, outs):
        assert p.returncode == 0, e
    recs = [json.loads(o.strip().splitlines()[-1]) for o, _ in outs]
    assert sorted(r["rank"] for r in recs) == [0, 1]
    assert all(r["world"] == 2 and r["max"] == 2.0 for r in recs)


def test_reference_arm_other_ranks_exit_without_work():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", CUDA_VISIBLE_DEVICES="")
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True, text=True,
                       timeout=120)
    assert p.returncode == 0 and p.stdout.strip() == ""
