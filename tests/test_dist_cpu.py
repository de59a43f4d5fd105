"""The multi-process (N > 1) paths on CPU with the gloo backend, world size 2.

Two multi-GPU modes: layers of a job are independent (each rank quantizes its own layer,
no data-path collective: the timing reduction, the per-rank inputs and the launch of both
benchmark arms under torch.distributed.run), and one layer sharded over the ranks
(paper_2607_07964_gb300.sharded: token-split factors with one all-reduce, row-split sweep
with one all-gather), whose partition and exchange logic runs here with the oracle as the
compute backend.
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


# ------------------------------------------------------------------ sharded single layer
class OracleBackend:
    """The sharded layer's stages through the oracle on CPU tensors (float64), so that the
    partition and the collectives of ShardedLayer run under gloo without a GPU."""

    def __init__(self, bits, group, block, damp):
        self.bits, self.group, self.block, self.damp = bits, group, block, damp

    def factor(self, A):
        from oracle import kronq_oracle as ref
        return torch.from_numpy(ref.accum_factor(A.numpy()))

    def stages_2_3(self, W, HX, HG, sign_u, sign_v):
        from oracle import kronq_oracle as ref
        b = ref.biip(W.numpy(), HX.numpy(), HG.numpy(), sign_u.numpy(), sign_v.numpy())
        R = ref.inverse_cholesky_upper(ref.damp(b["HX"], self.damp))
        return torch.from_numpy(b["W"]), torch.from_numpy(R)

    def sweep(self, Wp_rows, R):
        from oracle import kronq_oracle as ref
        o = ref.obs_sweep(Wp_rows.numpy(), R.numpy(), self.bits, self.group, self.block)
        return (torch.from_numpy(o["codes"]), torch.from_numpy(o["scale"]),
                torch.from_numpy(o["zero"]))


SHARD_CFG = dict(d_out=56, d_in=64, T=301, bits=3, group=32, block=32)


def _sharded_worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    from paper_2607_07964_gb300.sharded import ShardedLayer, split_range
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        c = SHARD_CFG
        cfg = kqsynth.CONFIGS["tiny256"].replace(d_out=c["d_out"], d_in=c["d_in"], T=c["T"], bits=c["bits"],
                                                 group=c["group"], n_outliers=2)
        L = kqsynth.layer(cfg)
        t0, t1 = split_range(c["T"], rank, world)
        layer = ShardedLayer(OracleBackend(c["bits"], c["group"], c["block"], 0.01))
        HX, HG = layer.factors(torch.from_numpy(L["X"][t0:t1]), torch.from_numpy(L["G"][t0:t1]))
        codes, scale, zero = layer.run(torch.from_numpy(L["X"][t0:t1]), torch.from_numpy(L["G"][t0:t1]),
                                       torch.from_numpy(L["W"]), torch.from_numpy(L["sign_u"]),
                                       torch.from_numpy(L["sign_v"]))
        # a ragged row count: 37 rows over the ranks, each rank's part tagged with its rows
        r0, r1 = split_range(37, rank, world)
        part = torch.arange(r0, r1, dtype=torch.int32)[:, None].repeat(1, 3)
        ragged = layer.gather_rows(part, 37)
        np.savez(os.path.join(out_dir, f"s{rank}.npz"), HX=HX.numpy(), HG=HG.numpy(), codes=codes.numpy(),
                 scale=scale.numpy(), zero=zero.numpy(), ragged=ragged.numpy(), tokens=np.array([t0, t1]))
    finally:
        torch.distributed.destroy_process_group()


def test_sharded_layer_token_split_and_row_split_gloo(tmp_path):
    """Per-rank token partial sums all-reduced equal the full factors; the row-split sweep
    gathered on every rank is the sweep of the whole layer on the same factors."""
    from oracle import kronq_oracle as ref
    port = _free_port()
    mp.start_processes(_sharded_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    res = [np.load(tmp_path / f"s{r}.npz") for r in range(2)]
    c = SHARD_CFG
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_out=c["d_out"], d_in=c["d_in"], T=c["T"], bits=c["bits"],
                                             group=c["group"], n_outliers=2)
    L = kqsynth.layer(cfg)
    # the two token ranges partition the tokens
    assert res[0]["tokens"][0] == 0 and res[0]["tokens"][1] == res[1]["tokens"][0] and res[1]["tokens"][1] == c["T"]
    for key, A in (("HX", L["X"]), ("HG", L["G"])):
        full = ref.accum_factor(A)
        for r in range(2):
            assert np.linalg.norm(res[r][key] - full) <= 1e-12 * np.linalg.norm(full)
        assert np.array_equal(res[0][key], res[1][key])       # every rank holds the same reduced factor
    # the whole layer swept on one process from the same reduced factors
    b = ref.biip(L["W"], res[0]["HX"], res[0]["HG"], L["sign_u"], L["sign_v"])
    R = ref.inverse_cholesky_upper(ref.damp(b["HX"], 0.01))
    want = ref.obs_sweep(b["W"], R, c["bits"], c["group"], c["block"])
    for r in range(2):
        # the dense fp64 products of stages 2-3 may round differently from one process to
        # another (threaded BLAS); codes and zero points are the same, grids to fp64 rounding
        assert np.array_equal(res[r]["codes"], want["codes"])
        assert np.allclose(res[r]["scale"], want["scale"], rtol=1e-12, atol=0)
        assert np.array_equal(res[r]["zero"], want["zero"])
        assert np.array_equal(res[r]["ragged"][:, 0], np.arange(37))
    assert np.array_equal(res[0]["codes"], res[1]["codes"])
