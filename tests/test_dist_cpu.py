"""The multi-process (N > 1) paths on CPU with the gloo backend, world size 2.

The layers of a job are independent (each rank quantizes its own layer, no data-path
collective), so the N > 1 logic is the timing reduction (the slowest rank's time), the
per-rank inputs, and the launch of both benchmark arms under torch.distributed.run.
"""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import kqsynth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import bench
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        got = bench.max_over_ranks(10.0 + 3.0 * rank, world)
        alone = bench.max_over_ranks(5.0, 1)
        with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
            json.dump({"max": got, "alone": alone}, f)
    finally:
        torch.distributed.destroy_process_group()


def test_max_over_ranks_gloo(tmp_path):
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    for r in range(2):
        res = json.load(open(tmp_path / f"r{r}.json"))
        assert res["max"] == 13.0       # every rank sees the slowest rank's time
        assert res["alone"] == 5.0


def test_ranks_get_independent_layers():
    """Weak scaling: rank r quantizes the layer drawn with seed r."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(T=64)
    a = kqsynth.layer(cfg.replace(seed=0))
    b = kqsynth.layer(cfg.replace(seed=1))
    assert not np.array_equal(a["X"], b["X"])
    assert not np.array_equal(a["W"], b["W"])
    c = kqsynth.layer(cfg.replace(seed=1))
    assert np.array_equal(b["X"], c["X"])


def test_reference_arm_under_torchrun():
    """bench.py --impl reference launched as the driver launches N > 1 jobs: rank 0 prints
    one JSON line, every rank exits 0."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--steps", "1", "--warmup", "0", "--config", "tiny256"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    out = json.loads(lines[0])
    assert out["impl"] == "reference" and out["n_gpus"] == 2
    assert out["value"] > 0 and out["unit"] == "ms" and out["higher_is_better"] is False
    assert out["cpu_baseline"]["kind"] == "oracle"
