"""The multi-process (one rank per GPU) path of bench.py on CPU with the gloo backend, world
size 2: the cross-rank aggregation of a weak-scaling run, and the reference arm launched by
torchrun (rank 0 alone runs and prints the JSON line; the other ranks exit 0 without work).
The data path has no collective: each rank quantizes its own matrix (seed + rank)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _aggregate_worker(rank, ws, port, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        # rank r ran for 10 (r + 1) ms and scored 100 (r + 1) pairs
        t, sc = bench.rank_aggregate(10.0 * (rank + 1), 100.0 * (rank + 1), ws,
                                     torch.device("cpu"))
        out[rank] = (t, sc)
    finally:
        dist.destroy_process_group()


def test_rank_aggregate_two_ranks_gloo():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_aggregate_worker, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0] == res[1] == (20.0, 300.0)  # slowest rank's time, all ranks' scores


def test_rank_aggregate_single_rank_is_identity():
    import bench
    assert bench.rank_aggregate(12.5, 7.0, 1, None) == (12.5, 7.0)


def test_reference_arm_under_torchrun_two_ranks():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--config",
           "c1", "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["scaling"] == "weak"
    assert d["value"] > 0 and d["e2e"]["value"] == d["value"]
    assert d["cpu_baseline"]["kind"] == "oracle"


def test_each_rank_quantizes_its_own_matrix():
    import numpy as np
    import synthetic as S
    cfg = S.C1
    w0 = S.gen_W(cfg.with_(seed=cfg.seed + 0), np.arange(4))
    w1 = S.gen_W(cfg.with_(seed=cfg.seed + 1), np.arange(4))
    assert w0.shape == w1.shape and not np.array_equal(w0, w1)

