"""Multi-process (world size 2) logic of bench.py on the CPU with the gloo backend.

Layers are independent, so the multi-GPU run gives each rank its own layer and
exchanges nothing on the data path; the only collectives are the reduction of the
timed figures (slowest rank's time, all ranks' keys).  These tests run that logic in
two real processes over gloo, and the reference arm under torch.distributed.run.
"""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    import synth
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        layer = bench.layer_of_rank(rank)
        # each rank times its own steps; the whole job is the slowest rank over all keys
        ms, keys = bench.reduce_over_ranks(10.0 + 5.0 * rank, 100.0 * (rank + 1), world, "cpu")
        wl = bench.make_workload("tiny_fp32_l1h2_d64", world)
        K, _ = synth.LayerRollout(wl, layer).block(0)
        q.put((rank, layer, ms, keys, wl.L, float(np.abs(K).sum()), bench.reference_runs_on(rank)))
    finally:
        dist.destroy_process_group()


def test_two_ranks_reduce_and_own_layers():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=240) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, l0, ms0, k0, L0, s0, ref0), (r1, l1, ms1, k1, L1, s1, ref1) = out
    assert (l0, l1) == (0, 1)                       # one layer per rank
    assert ms0 == ms1 == 15.0                       # the slowest rank's time
    assert k0 == k1 == 300.0                        # keys of all ranks
    assert L0 == L1 == 2                            # the workload grows to one layer per rank
    assert s0 != s1                                 # distinct synthetic streams per layer
    assert ref0 and not ref1                        # the reference arm runs on rank 0 only


def test_reference_arm_under_torchrun_prints_once():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--workload", "tiny_fp32_l1h2_d64", "--steps", "1",
           "--warmup", "3"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle"
