"""bench.py has no multi-GPU path: the attention kernels share key tiles among
the CTAs of a cluster by TMA multicast within one GPU's memory, which may only
run in single-GPU jobs. Under torchrun with two ranks (the environment a
2-GPU launch gives each process), rank 0 prints one "unavailable" line and
both ranks exit 0 without touching a GPU; neither initialises a process
group."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(rank, *args):
    env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2",
               MASTER_ADDR="127.0.0.1", MASTER_PORT="29999", CUDA_VISIBLE_DEVICES="")
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--gpus", "2", *args],
                          capture_output=True, text=True, env=env, cwd=ROOT, timeout=300)


def test_two_ranks_report_unavailable_and_exit_zero():
    r0, r1 = _run(0), _run(1)
    assert r0.returncode == 0 and r1.returncode == 0, (r0.stderr[-2000:], r1.stderr[-2000:])
    assert r1.stdout.strip() == ""
    lines = [l for l in r0.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["n_gpus"] == 2 and "multicast" in d["unavailable"]
    assert d["metric"].startswith("MLA attention")


def test_bench_source_has_no_collective():
    src = open(os.path.join(ROOT, "bench.py")).read()
    for word in ("nccl", "init_process_group", "all_reduce", "torch.distributed"):
        assert word not in src, word
