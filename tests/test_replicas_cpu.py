"""The replica path of a multi-GPU run, on CPU: two gloo ranks.  Sequences
are independent, so the ranks exchange nothing on the data path; the
barrier around the timed region, the maximum of the per-rank times, the
whole-job rate and each replica's own prompts are the multi-rank steps, and
the reference arm runs on rank 0 alone."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

pytest.importorskip("torch")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

WORKER = r"""
import json, os, sys
import torch.distributed as dist
rank, world = int(os.environ["RANK"]), int(os.environ["WORLD_SIZE"])
dist.init_process_group("gloo", rank=rank, world_size=world)
import bench
import workloads as wl
r = bench.Ranks(world, "cpu")
r.barrier()
ms = float(sys.argv[1].split(",")[rank])
mx = r.max(ms)
w = wl.get_workload("tiny")
p = bench.replica_prompts(w, rank)
r.barrier()
print(json.dumps({"rank": rank, "max_ms": mx, "rate": bench.whole_job_rate(world, w.batch * w.gen_len, 3, mx),
                  "prompts": p.tolist()}))
dist.destroy_process_group()
"""


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def run_ranks(code, args, world=2, timeout=120):
    port = free_port()
    procs = []
    for rank in range(world):
        env = dict(os.environ, MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                   LOCAL_RANK=str(rank), WORLD_SIZE=str(world), CUDA_VISIBLE_DEVICES="")
        procs.append(subprocess.Popen([sys.executable, *code, *args], cwd=ROOT, env=env, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True))
    outs = []
    for pr in procs:
        try:
            o, e = pr.communicate(timeout=timeout)
        except subprocess.TimeoutExpired:
            for q in procs:
                q.kill()
            raise
        assert pr.returncode == 0, e[-2000:]
        outs.append(o)
    return outs


def test_two_gloo_ranks_time_and_rate():
    """Both ranks see the slower rank's time; the whole-job rate counts both
    ranks' tokens over it; the replicas' prompts differ and rank 0 keeps the
    workload's own."""
    import workloads as wl
    outs = run_ranks(["-c", WORKER], ["120.5,181.25"])
    res = sorted((json.loads(o.strip().splitlines()[-1]) for o in outs), key=lambda d: d["rank"])
    w = wl.get_workload("tiny")
    assert [d["max_ms"] for d in res] == [181.25, 181.25]
    assert res[0]["rate"] == res[1]["rate"] == 2 * w.batch * w.gen_len * 3 / 0.18125
    p0, p1 = np.array(res[0]["prompts"]), np.array(res[1]["prompts"])
    assert p0.shape == p1.shape == (w.batch, w.prompt_len) and not np.array_equal(p0, p1)
    assert np.array_equal(p0, wl.make_prompts(w, seed=w.seed))


def test_reference_arm_runs_on_rank_zero_only():
    """Under torchrun the reference arm's other ranks exit 0 without work
    and print nothing."""
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2", CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                        "--warmup", "0"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_bench_spawns_its_own_ranks():
    """`bench.py --gpus 2` outside torchrun starts two local ranks itself
    (torch.distributed.run, rendezvous on 127.0.0.1).  Run end to end on CPU
    through the reference arm: rank 0 prints the one JSON line, rank 1 exits
    0 without work."""
    env = {k: v for k, v in os.environ.items() if k not in ("RANK", "LOCAL_RANK", "WORLD_SIZE", "MASTER_ADDR",
                                                             "MASTER_PORT")}
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                        "--warmup", "0", "--workload", "tiny", "--cpu-sample-seconds", "1"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["ms_per_step"] > 0 and line["extrapolated_generation_ms"] > 0


def test_bench_refuses_a_mismatched_world_size():
    """Under torchrun, --gpus must equal WORLD_SIZE; otherwise bench.py fails
    loudly before any work."""
    env = dict(os.environ, RANK="0", LOCAL_RANK="0", WORLD_SIZE="3", CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                        "--warmup", "0"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode != 0
    assert "WORLD_SIZE" in r.stderr


def test_rank_launch_command():
    import bench
    cmd = bench.rank_launch_command(4, ["--gpus", "4", "--steps", "3"], 29555)
    assert cmd[1:3] == ["-m", "torch.distributed.run"]
    assert "--nproc-per-node=4" in cmd and "--master-port=29555" in cmd
    assert cmd[cmd.index("--master-addr") + 1] == "127.0.0.1"
    assert cmd[-4:] == ["--gpus", "4", "--steps", "3"] and cmd[-5].endswith("bench.py")
