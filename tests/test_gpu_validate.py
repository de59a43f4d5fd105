"""GPU parity of the Prop. 2 / incoherence statistics (validate.py, kq_compute_scales_exp,
kq_biip_stats) against the oracle, and the exponent sweep of Prop. 2 through the whole CUDA
path: the output-side rescale (h/a)^alpha gives the smallest proxy loss at alpha = 1/4 on the
synthetic layers, as the oracle's own pipeline does, and each loss is within 1e-3 of the
oracle's."""
import numpy as np
import pytest
import torch

import kqsynth
from oracle import kronq_oracle as ref

pytestmark = pytest.mark.gpu

DEV = "cuda"
ALPHAS = [0.0, 0.125, 0.25, 0.375, 0.5]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()


def K():
    from paper_2607_07964_gb300 import kronq
    return kronq


def _dev(a, dt=None):
    t = torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    return t if dt is None else t.to(dt)


def _factors(L):
    X, G = _dev(L["X"], torch.bfloat16), _dev(L["G"], torch.bfloat16)
    d_in, d_out = L["X"].shape[1], L["G"].shape[1]
    HX = torch.empty((d_in, d_in), device=DEV)
    HG = torch.empty((d_out, d_out), device=DEV)
    K().kq_accum_factor(X, HX)
    K().kq_accum_factor(G, HG)
    return X, G, HX, HG


@pytest.mark.parametrize("ex,eg", [(0.25, 0.25), (0.25, 0.125), (0.375, 0.0), (0.5, 0.5)])
def test_scales_exponent_parity(ex, eg):
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_out=128, d_in=256, T=1024)
    L = kqsynth.layer(cfg)
    _, _, HX, HG = _factors(L)
    W = _dev(L["W"])
    sx, sg = torch.empty(256, device=DEV), torch.empty(128, device=DEV)
    K().kq_compute_scales_exp(W, HX, HG, sx, sg, ex, eg)
    want_x, want_g = ref.biip_scales_exp(L["W"], np.diag(HX.cpu().numpy()), np.diag(HG.cpu().numpy()), ex, eg)
    assert np.allclose(sx.cpu().numpy(), want_x, rtol=1e-6, atol=0)
    assert np.allclose(sg.cpu().numpy(), want_g, rtol=1e-6, atol=0)
    if ex == 0.25 and eg == 0.25:
        sx2, sg2 = torch.empty_like(sx), torch.empty_like(sg)
        K().kq_compute_scales(W, HX, HG, sx2, sg2)
        assert torch.equal(sx, sx2) and torch.equal(sg, sg2)


def test_biip_stats_parity():
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_out=224, d_in=512, T=2048)
    L = kqsynth.layer(cfg)
    _, _, HX, HG = _factors(L)
    W = _dev(L["W"])
    out = torch.empty(4, dtype=torch.float64, device=DEV)
    ws = torch.empty(K().kq_biip_stats_workspace(224, 512), dtype=torch.uint8, device=DEV)
    K().kq_biip_stats(W, HX, HG, out, ws)
    got = out.cpu().numpy()
    W64 = L["W"].astype(np.float64)
    cv_in, cv_out = ref.norm_cv(W64)
    hx, hg = np.diag(HX.cpu().numpy()), np.diag(HG.cpu().numpy())
    want = [cv_in, cv_out, ref.rho(hx, np.sum(W64 ** 2, axis=0)), ref.rho(hg, np.sum(W64 ** 2, axis=1))]
    assert np.allclose(got, want, rtol=1e-6, atol=0)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_prop2_exponent_sweep(seed):
    from paper_2607_07964_gb300.validate import exponent_sweep
    cfg = kqsynth.CONFIGS["tiny256"].replace(T=4096, seed=seed)
    L = kqsynth.layer(cfg)
    X, G = _dev(L["X"], torch.bfloat16), _dev(L["G"], torch.bfloat16)
    res = exponent_sweep(X, G, _dev(L["W"]), _dev(L["sign_u"], torch.int8), _dev(L["sign_v"], torch.int8), 3, 0,
                         ALPHAS)
    want = [ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], 3, 0, 128, 0.01, eg=a)["loss"]
            for a in ALPHAS]
    for g, w in zip(res["loss"], want):
        assert abs(g - w) <= 1e-3 * w
    assert ALPHAS[int(np.argmin(res["loss"]))] == 0.25
    st = res["stats"]
    # BiIP's output rotation mixes the rows: the row norms end up more even than after the
    # input side alone
    assert st["biip"]["cv_out"] < st["hx_only"]["cv_out"]
    assert 0.0 < st["rho_out"] < 1.0 and 0.0 < st["rho_in"] < 1.0
