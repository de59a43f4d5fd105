"""Checks of Proposition 2 and of the incoherence statistics on a layer, run through the CUDA
path: the output-side exponent sweep of the rescale (Prop. 2: s_i = (h_i / a_i)^alpha is best
at alpha = 1/4), Prop. 2's gain rho, and the coefficient of variation of the column and row
norms of W before, after input-side-only processing (S_X, V) and after BiIP (Sec. 3.2 and
the appendix on weight distributions). Only orders libkronq calls.
"""
from __future__ import annotations

import torch

from . import kronq as kq
from .pipeline import LayerPipeline


def biip_statistics(W, HX, HG, s_x, s_g, sign_u, sign_v, stream=None) -> dict:
    """CV_in / CV_out of W, of W S_X V^T (H_X-side only) and of U S_G W S_X V^T (BiIP), and
    rho_in / rho_out from the raw factors' diagonals. HX, HG raw; s_x, s_g the scales."""
    d_out, d_in = W.shape
    ws = torch.empty(kq.kq_biip_stats_workspace(d_out, d_in), dtype=torch.uint8, device=W.device)
    out = {}
    buf = torch.empty(4, dtype=torch.float64, device=W.device)
    kq.kq_biip_stats(W, HX, HG, buf, ws, stream=stream)
    torch.cuda.synchronize()
    v = buf.cpu().tolist()
    out["original"] = {"cv_in": v[0], "cv_out": v[1]}
    out["rho_in"], out["rho_out"] = v[2], v[3]
    Wx = W.clone()
    kq.kq_rotate_in(Wx, None, s_x, sign_v, kq.KQ_FWD, stream=stream)
    kq.kq_biip_stats(Wx, None, None, buf, ws, stream=stream)
    torch.cuda.synchronize()
    v = buf.cpu().tolist()
    out["hx_only"] = {"cv_in": v[0], "cv_out": v[1]}
    kq.kq_rotate_out(Wx, None, s_g, sign_u, kq.KQ_FWD, stream=stream)
    kq.kq_biip_stats(Wx, None, None, buf, ws, stream=stream)
    torch.cuda.synchronize()
    v = buf.cpu().tolist()
    out["biip"] = {"cv_in": v[0], "cv_out": v[1]}
    return out


def exponent_sweep(X, G, W, sign_u, sign_v, bits: int, group: int, alphas, block: int = 128,
                   damp: float = 0.01, trailing: str = "3xtf32") -> dict:
    """Proxy loss tr(H_G dW H_X dW^T) of the quantized layer for each output-side exponent
    alpha (S_X kept at 1/4), plus the statistics above at alpha = 1/4."""
    d_out, d_in = W.shape
    dev = W.device
    HX = torch.empty((d_in, d_in), device=dev)
    HG = torch.empty((d_out, d_out), device=dev)
    kq.kq_accum_factor(X, HX)
    kq.kq_accum_factor(G, HG)
    p = LayerPipeline(d_out, d_in, bits, group, block, damp, device=dev, want_col_loss=False, trailing=trailing,
                      g_chunk_tokens=0)
    What = torch.empty_like(W)
    loss = torch.zeros(1, dtype=torch.float64, device=dev)
    lws = torch.empty(kq.kq_proxy_loss_workspace(d_out, d_in), dtype=torch.uint8, device=dev)
    res = {"alphas": list(alphas), "loss": []}
    for a in alphas:
        kq.kq_compute_scales_exp(W, HX, HG, p.s_x, p.s_g, 0.25, a)
        kq.kq_traces(HX, p.s_x, HG, p.s_g, p.traces)
        p.run_from_factors(HX, HG, W, sign_u, sign_v, scales_ready=True)
        p.check()
        kq.kq_dequant_revert(p.codes, p.scale, p.zero, group, p.s_x, p.s_g, sign_u, sign_v, What)
        kq.kq_proxy_loss(W, What, HX, HG, loss, lws)
        torch.cuda.synchronize()
        res["loss"].append(float(loss.item()))
        if a == 0.25:
            res["stats"] = biip_statistics(W, HX, HG, p.s_x.clone(), p.s_g.clone(), sign_u, sign_v)
    return res
