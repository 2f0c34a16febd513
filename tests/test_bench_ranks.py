"""The benchmark's multi-process path on the CPU (the path runs independent
replicas, one per GPU, with no collective on the data path): under torchrun
with world size 2 (gloo), every rank takes the slowest replica's time and the
whole-job throughput counts every replica's work; the reference arm prints one
line from rank 0 and the other rank exits 0 without work."""
import json
import os
import socket
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _torchrun(args, timeout):
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(_free_port())] + args
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, r.stderr[-3000:]
    return [json.loads(ln) for ln in r.stdout.splitlines() if ln.strip().startswith("{")]


def test_replicas_take_the_slowest_rank_time():
    out = _torchrun([os.path.join("tests", "bench_rank_worker.py")], 300)
    assert len(out) == 1 and out[0]["world"] == 2
    ranks = sorted(out[0]["ranks"], key=lambda d: d["rank"])
    assert [d["rank"] for d in ranks] == [0, 1]
    assert all(d["slowest_ms"] == 15.0 for d in ranks)
    expect = 2 * 2.0e12 / 15e-3 / 1e12            # two replicas' operations over the slower one's step
    assert all(abs(d["tops"] - expect) <= 1e-9 * expect for d in ranks)


def test_reference_arm_under_torchrun_prints_from_rank_0_only():
    lines = _torchrun(["bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1"], 600)
    assert len(lines) == 1
    line = lines[0]
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["scaling"] == "weak"
    assert line["config"]["parallelism"] == "replicas2"
