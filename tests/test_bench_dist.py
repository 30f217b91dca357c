"""The multi-replica logic of bench.py on CPU: two gloo ranks (world size 2)
check that every time is the max over ranks, that the value counts all
ranks' work, and that the reference arm runs on rank 0 only."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

WORKER = r"""
import io, json, os, sys, contextlib
sys.path.insert(0, {root!r})
import torch.distributed as dist
dist.init_process_group("gloo")
import bench
rank, ws = dist.get_rank(), dist.get_world_size()
# rank r took (r + 1) * 10 ms on every phase
got = bench.reduce_max([10.0 * (rank + 1), 5.0 * (rank + 1)], "cpu")
rate = bench.job_rate(1e6, ws, 4, got[0])
# the reference arm: rank 0 alone runs and prints; the others exit quietly
buf = io.StringIO()
# one core: a spawned oracle pool would re-run this script's top level
args = type("A", (), dict(steps=1, warmup=0, ref_seconds=0.05, cpu_cores=1))()
with contextlib.redirect_stdout(buf):
    os.environ["RANK"], os.environ["WORLD_SIZE"] = str(rank), str(ws)
    bench.run_reference(args)
print(json.dumps({{"rank": rank, "got": got, "rate": rate, "ref": buf.getvalue()}}))
dist.destroy_process_group()
"""


def test_two_gloo_ranks(tmp_path):
    pytest.importorskip("torch")
    script = tmp_path / "worker.py"
    script.write_text(WORKER.format(root=ROOT))
    env = dict(os.environ, MASTER_ADDR="127.0.0.1", MASTER_PORT="29641", WORLD_SIZE="2")
    procs = []
    for r in range(2):
        procs.append(subprocess.Popen([sys.executable, str(script)], cwd=ROOT,
                                      env=dict(env, RANK=str(r), LOCAL_RANK=str(r)),
                                      stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=300)
        assert p.returncode == 0, err[-2000:]
        outs.append(json.loads(out.strip().splitlines()[-1]))
    outs.sort(key=lambda o: o["rank"])
    for o in outs:
        assert o["got"] == [20.0, 10.0]                 # the slowest rank's times
        assert o["rate"] == pytest.approx(2 * 1e6 * 4 / 0.020)  # both ranks' work
    line = json.loads(outs[0]["ref"].strip())
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0
    assert outs[1]["ref"] == ""


def test_reference_arm_on_several_host_cores():
    """The reference arm as the driver launches it: the unchanged oracle in
    two spawned processes; the line reports the cores it used and the
    single-process rate beside the total."""
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "0", "--ref-seconds", "0.5",
                          "--cpu-cores", "2"],
                         cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0
    cb = line["cpu_baseline"]
    assert cb["cores"] == 2 and cb["kind"] == "oracle"
    assert 0 < cb["single_core_value"] <= cb["value"] * 1.01
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
