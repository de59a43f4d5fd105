"""The debug build (libkronq_debug.so, -DKQ_DEBUG): the kernels check every store index
against the size of the buffer it belongs to and record a failed check instead of
faulting (a stand-in for a memory checker, which is closed on this machine).

  * the self-test's out-of-range index is caught, skipped and reported with its source
    file and line; the normal build has no checks and reports nothing;
  * whole layers through the debug build (two-stream schedule, both trailing-update modes,
    ragged and large-layer shapes, the drift correction, decode) record no failed check
    and give the same bits as the normal build.
Runs in child processes, since a process loads one of the two libraries.
"""
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import hashlib, json, os, sys
import numpy as np, torch
sys.path.insert(0, os.environ["KQ_ROOT"])
import kqsynth
from paper_2607_07964_gb300 import kronq as K
from paper_2607_07964_gb300.pipeline import LayerPipeline
out = {"debug": K.kq_debug_build()}
buf = torch.zeros(1001, device="cuda")
K.kq_selftest_bounds(buf, 1000)
out["selftest"] = K.kq_debug_status()
out["selftest_last"] = float(buf[1000])
res = {}
for name, over, trailing, drift in [
        ("a", dict(d_out=512, d_in=1792, bits=3, group=128, T=2048), "3xtf32", None),
        ("b", dict(d_out=7168, d_in=3584, bits=4, group=0, T=1024), "3xtf32", None),
        ("c", dict(d_out=448, d_in=896, bits=2, group=128, T=1000), "fp32", None),
        ("d", dict(d_out=256, d_in=1024, bits=4, group=128, T=2048), "3xtf32", 0.25)]:
    cfg = kqsynth.CONFIGS["tiny256"].replace(w_bf16=True, **over)
    L = kqsynth.layer(cfg)
    dev = lambda a, dt=torch.float32: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(dt)
    args = (dev(L["X"], torch.bfloat16), dev(L["G"], torch.bfloat16), dev(L["W"]),
            dev(L["sign_u"], torch.int8), dev(L["sign_v"], torch.int8))
    p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, trailing=trailing,
                      alpha=drift)
    Xt = dev(kqsynth.fp_activations(cfg, L["X"]), torch.bfloat16) if drift else None
    p.run(*args, Xt=Xt)
    p.check()
    digest = lambda t: hashlib.sha256(t.cpu().numpy().tobytes()).hexdigest()
    res[name] = {k: digest(getattr(p, k)) for k in ("codes", "scale", "zero", "Lt")}
    if name == "a":
        packed = torch.empty(K.kq_packed_codes_bytes(cfg.d_out, cfg.d_in, cfg.bits) // 4, dtype=torch.int32,
                             device="cuda")
        K.kq_pack_codes(p.codes, cfg.bits, packed)
        x = torch.randn((2, cfg.d_in), device="cuda", generator=torch.Generator("cuda").manual_seed(1))
        y = torch.empty((2, cfg.d_out), device="cuda")
        ws = torch.empty(K.kq_infer_workspace(2, cfg.d_in, cfg.d_out), dtype=torch.uint8, device="cuda")
        info = torch.zeros(1, dtype=torch.int32, device="cuda")
        K.kq_infer(packed, p.scale, p.zero, cfg.d_out, cfg.d_in, cfg.bits, cfg.group, p.s_x, p.s_g,
                   args[3], args[4], x, y, ws, info=info)
        assert K.kq_check(info)[0] == K.KQ_OK
        res[name]["y"] = digest(y)
out["layers"] = res
out["after"] = K.kq_debug_status()
print(json.dumps(out))
'''


def _child(debug: bool) -> dict:
    import json
    env = dict(os.environ, KQ_ROOT=ROOT, KQ_DEBUG="1" if debug else "0")
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stderr[-3000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_debug_build_catches_bounds_and_agrees_with_normal_build():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()
    build.build(debug=True)
    dbg = _child(True)
    rel = _child(False)
    assert dbg["debug"] == 1 and rel["debug"] == 0
    # the self-test's index n is caught in the debug build (file "api"), not written
    assert dbg["selftest"][0] == "api" and dbg["selftest"][1] > 0
    assert dbg["selftest_last"] == 0.0
    # the normal build has no checks: nothing recorded, and the (in-bounds) write happened
    assert rel["selftest"] == [None, 0] and rel["selftest_last"] == 1000.0
    # no failed check anywhere in the layers, and the same results
    assert dbg["after"] == [None, 0], dbg["after"]
    assert dbg["layers"] == rel["layers"]
