"""The multi-rank product path on the GPU: bench.py's own shard code run as
two ranks (two processes on GPU 0, each committing its contiguous half of
the ragged 152M-element shard c3 under the flat-parameter partition,
--split model), with the post-step exchange through cohort.agree over Gloo.
The ranks never wait on each other's kernels, only on the host control
plane.  The whole-model digests of the two ranks must equal a single
process's over the whole workload, and the first step's must equal the
oracle's (the digest of a concatenation is the sum of the digests)."""
import json
import os
import socket
import subprocess
import sys

import pytest

from apc_testlib import oracle_workload_digest
from synth import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # the CUDA path has no fallback: without a GPU these tests cannot run
    pytest.skip("no CUDA device", allow_module_level=True)

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ARGS = ["--workload", "c3", "--split", "model", "--steps", "2", "--warmup", "3", "--no-e2e", "--no-cpu-baseline",
        "--no-clocks", "--no-next"]


def run_ranks(world: int) -> dict:
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    procs = []
    for r in range(world):
        env = dict(os.environ, RANK=str(r), WORLD_SIZE=str(world), LOCAL_RANK="0", LOCAL_WORLD_SIZE=str(world),
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        procs.append(subprocess.Popen([sys.executable, os.path.join(ROOT, "bench.py"), "--gpus", str(world)] + ARGS,
                                      env=env, cwd=ROOT, stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = []
    try:
        for p in procs:
            outs.append(p.communicate(timeout=900))
    finally:
        for p in procs:
            if p.poll() is None:
                p.kill()
    for p, (out, err) in zip(procs, outs):
        assert p.returncode == 0, err[-3000:]
    lines = [x for x in outs[0][0].splitlines() if x.startswith("{")]
    assert len(lines) == 1 and not any(x.startswith("{") for o, _ in outs[1:] for x in o.splitlines())  # rank 0 alone prints the line
    return json.loads(lines[0])


def test_two_rank_model_split_equals_one_process_and_oracle():
    one, two = run_ranks(1), run_ranks(2)
    assert two["n_gpus"] == 2 and two["config"]["split"] == "model" and two["scaling"] == "strong"
    assert two["config"]["elements"] == one["config"]["elements"] == W.c3().n
    assert two["config"]["elements_per_rank"] == W.c3().n // 2
    assert one["verify_matches_commit"] and two["verify_matches_commit"]
    assert two["first_commit_digests"] == one["first_commit_digests"]
    assert two["digests"] == one["digests"]
    want = oracle_workload_digest(W.c3(), 10)
    assert one["first_commit_digests"] == ["%016x" % d for d in want]
