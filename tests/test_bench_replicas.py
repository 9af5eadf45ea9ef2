"""The benchmark's multi-process path on the CPU (gloo, world size 2).

`bench.py --gpus N` runs N independent replicas under torchrun (weak scaling): each rank
decodes its own seeded prompt, and the ranks meet only in a barrier around the timed region
and a max-reduce of the timings.  These tests run that host logic as two gloo processes, and
the CPU reference arm as a two-rank torchrun job whose rank 0 alone prints the line.
"""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_RANK_SCRIPT = r"""
import argparse, hashlib, json, sys
sys.path.insert(0, {root!r})
import bench
import dllm_inputs as I
args = argparse.Namespace(impl="reference")
world, rank, local, pg = bench._dist_setup(args)
assert pg is not None and world == 2 and local == rank, (world, rank, local)
bench._barrier(pg)
mx = bench._max_over_ranks(10.0 + rank, pg)
prompt = I.uniform_prompt(bench.LP, bench.SHAPE["vocab"], bench.SHAPE["mask_id"], seed=I.SEED_PROMPT + rank)
digest = hashlib.sha256(prompt.tobytes()).hexdigest()
gathered = [None, None]
pg.all_gather_object(gathered, digest)
bench._barrier(pg)
pg.destroy_process_group()
print(json.dumps({{"rank": rank, "max": mx, "digests": gathered}}))
"""


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_replica_ranks_meet_only_in_barrier_and_max():
    port = _free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2", MASTER_ADDR="127.0.0.1",
                   MASTER_PORT=str(port))
        procs.append(subprocess.Popen([sys.executable, "-c", _RANK_SCRIPT.format(root=ROOT)], env=env, cwd=ROOT,
                                      stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=180)
        assert p.returncode == 0, err[-2000:]
        outs.append(json.loads(out.strip().splitlines()[-1]))
    for o in outs:
        assert o["max"] == 11.0  # the max over ranks, seen by every rank
        d0, d1 = o["digests"]
        assert d0 != d1  # each replica decodes its own prompt
    assert outs[0]["digests"] == outs[1]["digests"]


def test_reference_arm_two_ranks_prints_one_line():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
           "--warmup", "0"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


if __name__ == "__main__":
    sys.exit(pytest.main([__file__, "-q"]))
