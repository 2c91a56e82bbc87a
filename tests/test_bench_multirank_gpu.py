"""bench.py's multi-rank path on the GPU: two ranks under torchrun, both on
cuda:0, exchanging their histograms (Algorithm 1 steps 2 and 5) through
gloo, which goes through host memory.  This runs the library's multi-rank
calling pattern (per-pass calls, the summed [E,256] counts, the global
target rank) and checks that every rank forms the same next bias.  It is
not a scaling measurement: each box here has one GPU."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = pytest.mark.gpu


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("workload,tokens", [("global", 131072), ("tie", 65536), ("router", 65536)])
def test_two_ranks_on_one_gpu_agree(cuda_ok, workload, tokens):
    env = dict(os.environ, EQB_BENCH_BACKEND="gloo", EQB_BENCH_DEVICE="0")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--gpus", "2", "--workload", workload, "--tokens", str(tokens),
           "--steps", "2", "--warmup", "3", "--e2e-steps", "0", "--no-cpu-baseline", "--no-extras"]
    out = subprocess.run(cmd, env=env, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["n_gpus"] == 2 and d["config"]["parallelism"] == "dp2"
    assert d["schedule"] == "per-pass calls, histograms all-reduced"
    assert d["ranks_agree"] is True
    assert d["value"] > 0 and d["scaling"] == "weak"
