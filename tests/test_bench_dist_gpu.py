"""bench.py under torchrun with two ranks, both on this machine's one GPU (gloo
carries the barrier and the max-reduce of the timings; the ranks' kernels
never wait on each other): one JSON line from rank 0 with the whole-job
figures, for the softmax line, the batched product and the long rows."""
import json
import os
import socket
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _torchrun(*args):
    env = dict(os.environ, BSM_BENCH_DIST_BACKEND="gloo")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py", "--gpus", "2",
           *args]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout[-3000:]
    return json.loads(lines[0])


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()


def test_softmax_line_two_ranks():
    d = _torchrun("--steps", "50", "--warmup", "3", "--e2e-steps", "2", "--no-cpu-baseline")
    assert d["n_gpus"] == 2 and d["value"] > 0 and d["device_status"] == 0
    assert d["config"]["parallelism"].startswith("2 ranks")
    assert d["e2e"]["value"] > 0 and d["gpu_launches"] == 50


def test_bmm_and_long_row_lines_two_ranks():
    d = _torchrun("--bmm", "2", "--steps", "50", "--warmup", "3", "--no-cpu-baseline")
    assert d["n_gpus"] == 2 and d["value"] > 0 and d["device_status"] == 0
    d = _torchrun("--long-rows", "65536", "--steps", "5", "--warmup", "3")
    assert d["n_gpus"] == 2 and d["value"] > 0 and d["device_status"] == 0
