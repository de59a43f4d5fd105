"""Failure behaviour without a GPU fault, and out-of-bounds writes caught by canaries.

  * NaN or Inf in an input never faults, and each case ends in a defined status. In the
    activations X the non-finite values spread to the rotated H_X, whose inverse Cholesky
    meets a pivot that is not positive: KQ_ERR_NOT_PD through the device error word. A NaN
    weight gives its column the dead-channel scale 1 and reaches the quantizer through W':
    KQ_ERR_NONFINITE; an infinite one gives the column scale 0, S_X^-1 makes H_X'
    non-finite: KQ_ERR_NOT_PD. In the gradients G they reach only S_G, where the
    channel gets the dead-channel scale 1: no status, finite codes. The context keeps
    working (a clean layer afterwards is correct).
  * Canary words: every buffer the layer reads or writes (inputs, outputs, factors, the
    Cholesky and sweep workspaces, the error words) sits inside a larger allocation whose
    guard regions before and after hold a fixed pattern; after whole layers (two-stream
    schedule and a CUDA graph replay) every guard still holds it.
(A stand-in for compute-sanitizer's memcheck, which is closed on this machine.)
"""
import numpy as np
import pytest
import torch

import kqsynth

pytestmark = pytest.mark.gpu

GUARD_BYTES = 4096
PATTERN = 0x5A


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()


def K():
    from paper_2607_07964_gb300 import kronq
    return kronq


def _cfg():
    return kqsynth.CONFIGS["tiny256"].replace(d_out=512, d_in=1792, bits=3, group=128, T=2048, w_bf16=True)


def _inputs(cfg, seed=0):
    L = kqsynth.layer(cfg.replace(seed=seed))
    dev = lambda a, dt=torch.float32: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(dt)  # noqa: E731
    return {"X": dev(L["X"], torch.bfloat16), "G": dev(L["G"], torch.bfloat16), "W": dev(L["W"]),
            "sign_u": dev(L["sign_u"], torch.int8), "sign_v": dev(L["sign_v"], torch.int8)}


def _run(p, inp):
    p.run(inp["X"], inp["G"], inp["W"], inp["sign_u"], inp["sign_v"])


@pytest.mark.parametrize("where,value", [("X", float("nan")), ("G", float("nan")), ("W", float("nan")),
                                         ("X", float("inf")), ("W", float("-inf"))])
def test_non_finite_input_reports_not_pd_and_context_survives(where, value):
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    cfg = _cfg()
    inp = _inputs(cfg)
    bad = dict(inp)
    bad[where] = inp[where].clone()
    bad[where][3, 5] = value
    p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp)
    _run(p, bad)
    torch.cuda.synchronize()
    if where == "G":
        # H_G reaches the sweep only through S_G, and a channel whose diagonal entry is not
        # a positive number gets the dead-channel scale 1: no status, no fault, finite codes
        p.check()
        assert float(p.s_g[5]) == 1.0
        assert torch.isfinite(p.scale).all()
    else:
        with pytest.raises(K().KronqError) as e:
            p.check()
        # X: H_X' is not finite and its Cholesky reports the pivot. W = NaN: the column's
        # norm is NaN, its scale the dead-channel 1, and the NaN reaches the quantizer through
        # W', which says so. W = -inf: the column's norm is +inf, its scale 0, and S_X^-1 makes
        # H_X' non-finite: the pivot again.
        want = K().KQ_ERR_NONFINITE if (where == "W" and value != value) else K().KQ_ERR_NOT_PD
        assert e.value.status == want, e.value
    # the same pipeline on clean inputs afterwards: no error, finite grids
    _run(p, inp)
    p.check()
    assert torch.isfinite(p.scale).all()
    assert torch.isfinite(p.Lt).all()


def _guarded(t: torch.Tensor) -> tuple[torch.Tensor, torch.Tensor]:
    """A copy of t inside an allocation with GUARD_BYTES of PATTERN before and after; returns
    (view, whole allocation as bytes)."""
    nbytes = t.numel() * t.element_size()
    whole = torch.full((GUARD_BYTES + nbytes + GUARD_BYTES,), PATTERN, dtype=torch.uint8, device=t.device)
    view = whole[GUARD_BYTES:GUARD_BYTES + nbytes].view(t.dtype).view(t.shape)
    view.copy_(t)
    return view, whole


def _guards_intact(whole: torch.Tensor) -> bool:
    return bool((whole[:GUARD_BYTES] == PATTERN).all()) and bool((whole[-GUARD_BYTES:] == PATTERN).all())


@pytest.mark.parametrize("trailing", ["3xtf32", "fp32"])
def test_canaries_around_every_buffer(trailing):
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    cfg = _cfg()
    inp = _inputs(cfg)
    p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, trailing=trailing)
    _run(p, inp)                       # one plain run first (one-time set-up), then guard everything
    p.check()
    want = {k: getattr(p, k).clone() for k in ("codes", "scale", "zero", "Lt")}
    wholes = {}
    for k in ("X", "G", "W", "sign_u", "sign_v"):
        inp[k], wholes["in." + k] = _guarded(inp[k])
    for k in ("HX", "HG", "Wp", "s_x", "s_g", "Lt", "codes", "scale", "zero", "col_loss", "traces", "trace_x",
              "trace_g", "info", "ws_chol", "ws_obs"):
        v, w = _guarded(getattr(p, k))
        setattr(p, k, v)
        wholes[k] = w
    _run(p, inp)
    p.check()
    graph, _ = p.capture(inp["X"], inp["G"], inp["W"], inp["sign_u"], inp["sign_v"])
    graph.replay()
    torch.cuda.synchronize()
    p.check()
    bad = [k for k, w in wholes.items() if not _guards_intact(w)]
    assert not bad, f"guard words overwritten around {bad}"
    for k, v in want.items():
        assert torch.equal(getattr(p, k), v), k
