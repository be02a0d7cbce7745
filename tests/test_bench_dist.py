"""bench.py's multi-process plumbing on CPU (gloo, world size 2).

Under torchrun each rank runs its own replica (replicas only: no collective on the data path);
the ranks meet at barriers and rank 0 reports the slowest rank's time.  These tests run the same
helpers bench.py uses, and the reference arm end to end, on two CPU processes.
"""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, ws, port, out):
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(ws), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    got_ws, got_rank, _ = bench.dist_init()
    assert (got_ws, got_rank) == (ws, rank)
    assert dist.get_backend() == "gloo"
    bench.barrier(ws)
    out[rank] = bench.max_over_ranks(ws, 10.0 * (rank + 1))   # slowest rank's time
    bench.barrier(ws)
    dist.destroy_process_group()


def test_ranks_meet_and_report_the_slowest_time():
    ws, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        procs = [ctx.Process(target=_rank, args=(r, ws, port, out)) for r in range(ws)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        assert dict(out) == {0: 20.0, 1: 20.0}


def test_reference_arm_under_torchrun_prints_one_line_from_rank_0():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--steps", "1", "--warmup", "0", "--workload", "tiny"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
    # the same workload keys as the GPU arm's config
    import synth
    spec = synth.SPECS["tiny"]
    sh = spec.shape
    want = {"workload": "tiny", "senders": spec.n_senders, "T": list(spec.T[:3]), "m": spec.m,
            "n_layers": sh.n_layers, "q_heads": sh.n_q_heads, "kv_heads": sh.n_kv_heads, "head_dim": sh.head_dim,
            "keep": spec.keeps[0]}
    assert {k: d["config"][k] for k in want} == want
