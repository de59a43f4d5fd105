"""GPU parity at the benchmark's full size: the Llama-3-8B q_proj layer (W 4096 x 4096,
T = 131072 calibration tokens, 4-bit, group 128), run through the same pipeline and the
same kernels the benchmark times. The oracle cannot redo the whole layer in float64 here,
so it checks what it can compute one by one:
  * sampled entries and the whole diagonal of H_X and H_G (float64 dot products);
  * S_X, S_G from those float64 diagonals;
  * sampled rows of W' = U S_G W S_X V^T (dense float64 products);
  * a 4096 x 4096 inverse Cholesky of an oracle-built SPD matrix;
  * the 4096 x 4096 sweep, bit-exact against the fp32-ordered oracle on sampled rows.
Inputs are drawn on the GPU with torch's generator (kqsynth.device_layer) and copied to
the host for the oracle.
"""
import numpy as np
import pytest
import torch

import kqsynth
from oracle import kronq_oracle as ref
from oracle import obs_sweep_fp32

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


@pytest.fixture(scope="module")
def layer():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()
    cfg = kqsynth.CONFIGS["q_proj_8b"]
    return cfg, kqsynth.device_layer(cfg)


def test_fullsize_factors_scales_rotation(layer):
    from paper_2607_07964_gb300 import kronq as K
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    cfg, inp = layer
    X, G, W = inp["X"], inp["G"], inp["W"]
    su, sv = inp["sign_u"], inp["sign_v"]
    d_out, d_in = cfg.d_out, cfg.d_in
    # the factors, as the pipeline's first stage computes them
    HX = torch.empty((d_in, d_in), device="cuda")
    HG = torch.empty((d_out, d_out), device="cuda")
    K.kq_accum_factor(X, HX)
    K.kq_accum_factor(G, HG)
    Xh = X.cpu().view(torch.int16).numpy()
    Gh = G.cpu().view(torch.int16).numpy()
    to32 = lambda a: (a.astype(np.uint32) << 16).view(np.float32)  # noqa: E731  bf16 bits -> fp32
    rng = np.random.default_rng(5)
    diags = []
    for A_bits, H, d in ((Xh, HX, d_in), (Gh, HG, d_out)):
        cols = np.unique(rng.integers(0, d, 48))
        A = to32(A_bits[:, cols].astype(np.uint16))
        pairs = [(a, b) for a in range(len(cols)) for b in range(len(cols))]
        want = ref.factor_entries(A, pairs).reshape(len(cols), len(cols))
        got = H.cpu().numpy()[np.ix_(cols, cols)]
        assert _rel(got, want) <= 1e-5
        diag_want = np.zeros(d)
        for t0 in range(0, A_bits.shape[0], 16384):   # float64 sums of squares over all tokens
            diag_want += ref.factor_diag(to32(A_bits[t0:t0 + 16384].view(np.uint16)))
        diag_got = torch.diagonal(H).cpu().numpy()
        assert np.max(np.abs(diag_got - diag_want) / diag_want) <= 1e-5
        diags.append(diag_want)
    hx, hg = diags
    # scales and the rotated weight, through the pipeline's own buffers
    p = LayerPipeline(d_out, d_in, cfg.bits, cfg.group, cfg.block, cfg.damp)
    K.kq_compute_scales(W, HX, HG, p.s_x, p.s_g)
    Wh = W.cpu().numpy().astype(np.float64)
    sx, sg = ref.biip_scales_from_diag(Wh, hx, hg)
    assert np.max(np.abs(p.s_x.cpu().numpy() / sx - 1)) <= 1e-5
    assert np.max(np.abs(p.s_g.cpu().numpy() / sg - 1)) <= 1e-5
    Wp = W.clone()
    K.kq_rotate_in(Wp, None, p.s_x, sv)
    K.kq_rotate_out(Wp, None, p.s_g, su)
    V = ref.rht_matrix(d_in, sv.cpu().numpy())
    U = ref.rht_matrix(d_out, su.cpu().numpy())
    M = (Wh * sx[None, :]) @ V.T
    rows = np.unique(rng.integers(0, d_out, 16))
    want = (U[rows] * sg[None, :]) @ M
    assert _rel(Wp.cpu().numpy()[rows], want) <= 1e-5


def test_fullsize_chol_and_sweep():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    from paper_2607_07964_gb300 import kronq as K
    build.build()
    n = 4096
    H = kqsynth.random_spd(n, seed=23, cond_decay=1.0).astype(np.float32)
    Lref = ref.lower_factor(ref.damp(H.astype(np.float64), 0.01))
    Lt = torch.empty((n, n), device="cuda")
    info = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(K.kq_chol_inv_workspace(n), dtype=torch.uint8, device="cuda")
    K.kq_chol_inv(torch.from_numpy(H).cuda(), 0.01, Lt, info, ws)
    assert K.kq_check(info)[0] == K.KQ_OK
    assert _rel(Lt.cpu().numpy(), Lref) <= 1e-5
    # the sweep on the oracle's L and a seeded W' of the q_proj size
    Lt32 = np.ascontiguousarray(Lref.astype(np.float32))
    gen = torch.Generator(device="cuda")
    gen.manual_seed(99)
    Wp = (0.05 * torch.randn((n, n), generator=gen, device="cuda")).contiguous()
    Wh = Wp.cpu().numpy()
    codes = torch.empty((n, n), dtype=torch.uint8, device="cuda")
    scale = torch.empty((n, n // 128), device="cuda")
    zero = torch.empty((n, n // 128), dtype=torch.int32, device="cuda")
    wso = torch.empty(K.kq_obs_quantize_workspace(n, n, 128), dtype=torch.uint8, device="cuda")
    K.kq_obs_quantize(Wp, torch.from_numpy(Lt32).cuda(), 4, 128, 128, codes, scale, zero, None, None, wso)
    rows = np.unique(np.random.default_rng(7).integers(0, n, 48))
    c = obs_sweep_fp32(Wh, Lt32, 4, 128, 128, rows=rows)
    assert np.array_equal(codes.cpu().numpy()[rows], c["codes"])
    assert np.array_equal(scale.cpu().numpy()[rows], c["scale"])
    assert np.array_equal(zero.cpu().numpy()[rows], c["zero"].astype(np.int32))
