"""GPU parity at full size for every Llama-shaped layer of the benchmark plan (q_proj and
the MLP layers of the 8B model; q/o, k/v and down_proj of the 70B model), each run through
the kernels and launch configuration the benchmark times (one H_X call, H_G in the
pipeline's token chunks). The oracle cannot redo these layers in float64, so it checks what
it can compute one by one, or what holds at any size:
  * sampled entries and sampled diagonal entries of H_X and H_G (float64 dot products over
    all T tokens);
  * S_X, S_G at the sampled channels;
  * sampled entries of W' = U S_G W S_X V^T and of H_X' = V S_X^-1 H_X S_X^-1 V^T (rows of
    U and V built one at a time from the Hadamard definition);
  * the inverse Cholesky: its trailing 1024 x 1024 block depends only on the trailing block
    of the damped H_X' (H = U U^T with U upper gives L = U^-T block by block), which the
    oracle factors exactly; and L L^T H e_j = e_j on sampled columns;
  * the sweep on the GPU's own W' and L, bit-exact against the fp32-ordered oracle on
    sampled rows.
Inputs are drawn on the GPU with torch's generator (kqsynth.device_layer).
"""
import numpy as np
import pytest
import torch

import kqsynth
from oracle import kronq_oracle as ref
from oracle import obs_sweep_fp32

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

CONFIGS = ["q_proj_8b", "gate_up_8b", "down_8b", "qo_70b", "kv_70b", "down_70b"]
TAIL = 1024


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _bf16_cols(A, cols):
    """float64 copy of the selected columns of a bf16 device matrix (exact widening)."""
    return A[:, torch.as_tensor(cols, device=A.device)].float().cpu().numpy().astype(np.float64)


@pytest.fixture(scope="module", params=CONFIGS)
def layer(request):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    from paper_2607_07964_gb300 import kronq as K
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    build.build()
    cfg = kqsynth.CONFIGS[request.param]
    inp = kqsynth.device_layer(cfg)
    d_out, d_in = cfg.d_out, cfg.d_in
    p = LayerPipeline(d_out, d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, overlap=False)
    s = torch.cuda.current_stream()
    # stage 1 as the pipeline launches it
    p._factor("X", inp["X"], p.HX, p.trace_x, p.info[0:1], s)
    p._factor("G", inp["G"], p.HG, p.trace_g, p.info[2:3], s)
    HX_raw = p.HX.clone()
    HG_raw = p.HG.clone()
    K.kq_compute_scales(inp["W"], p.HX, p.HG, p.s_x, p.s_g)
    p.Wp.copy_(inp["W"])
    K.kq_rotate_in(p.Wp, p.HX, p.s_x, inp["sign_v"], K.KQ_FWD)
    K.kq_rotate_out(p.Wp, None, p.s_g, inp["sign_u"], K.KQ_FWD)
    Wp = p.Wp.clone()
    K.kq_chol_inv(p.HX, cfg.damp, p.Lt, p.info[1:2], p.ws_chol)
    K.kq_obs_quantize(p.Wp, p.Lt, cfg.bits, cfg.group, cfg.block, p.codes, p.scale, p.zero, None, None, p.ws_obs)
    p.check()
    yield cfg, inp, p, HX_raw, HG_raw, Wp
    del p, inp, HX_raw, HG_raw, Wp
    torch.cuda.empty_cache()


def test_fullsize_factors_and_scales(layer):
    cfg, inp, p, HX, HG, _ = layer
    rng = np.random.default_rng(5)
    W = inp["W"].cpu().numpy().astype(np.float64)
    for A, H, d, s_dev, axis in ((inp["X"], HX, cfg.d_in, p.s_x, 0), (inp["G"], HG, cfg.d_out, p.s_g, 1)):
        cols = np.unique(rng.integers(0, d, 40))
        Ac = _bf16_cols(A, cols)
        want = Ac.T @ Ac                              # float64 sums over all tokens
        got = H[torch.as_tensor(cols, device="cuda")][:, torch.as_tensor(cols, device="cuda")].cpu().numpy()
        assert _rel(got, want) <= 1e-5
        assert np.max(np.abs(np.diag(got) / np.diag(want) - 1)) <= 1e-5
        # scales at these channels: (h / ||W column or row||^2)^(1/4)
        norm2 = np.sum(W[:, cols] ** 2, axis=0) if axis == 0 else np.sum(W[cols] ** 2, axis=1)
        s_want = (np.diag(want) / norm2) ** 0.25
        assert np.max(np.abs(s_dev.cpu().numpy()[cols] / s_want - 1)) <= 1e-5


def test_fullsize_rotations(layer):
    cfg, inp, p, HX, _, Wp = layer
    rng = np.random.default_rng(6)
    d_out, d_in = cfg.d_out, cfg.d_in
    sx = p.s_x.cpu().numpy().astype(np.float64)
    sg = p.s_g.cpu().numpy().astype(np.float64)
    su, sv = inp["sign_u"].cpu().numpy(), inp["sign_v"].cpu().numpy()
    rows = np.unique(rng.integers(0, d_out, 12))
    cols = np.unique(rng.integers(0, d_in, 12))
    U = ref.rht_rows(d_out, su, rows)
    V = ref.rht_rows(d_in, sv, cols)
    W = inp["W"].cpu().numpy().astype(np.float64)
    want = ((U * sg[None, :]) @ W * sx[None, :]) @ V.T
    got = Wp.cpu().numpy()[np.ix_(rows, cols)]
    assert _rel(got, want) <= 1e-5
    # H_X' = V S_X^-1 H_X S_X^-1 V^T at sampled entries
    hrows = np.unique(rng.integers(0, d_in, 12))
    Hh = HX.cpu().numpy().astype(np.float64)
    Vr = ref.rht_rows(d_in, sv, hrows) / sx[None, :]
    Vc = V / sx[None, :]
    want = (Vr @ Hh) @ Vc.T
    got = p.HX.cpu().numpy()[np.ix_(hrows, cols)]
    assert _rel(got, want) <= 1e-5


def test_fullsize_inverse_cholesky(layer):
    cfg, _, p, _, _, _ = layer
    n = cfg.d_in
    Hrot = p.HX.cpu().numpy().astype(np.float64)
    delta = cfg.damp * np.mean(np.diag(Hrot))
    L = p.Lt.cpu().numpy()
    # trailing block: exact against the oracle's inverse Cholesky of the damped trailing block
    D = Hrot[n - TAIL:, n - TAIL:] + delta * np.eye(TAIL)
    Lref = ref.lower_factor(D)
    assert _rel(L[n - TAIL:, n - TAIL:], Lref) <= 1e-5
    if n <= 4096:   # small enough for the whole float64 factor
        assert _rel(L, ref.lower_factor(ref.damp(Hrot, cfg.damp))) <= 1e-5
    assert np.all(np.triu(L, 1) == 0)
    # L L^T H e_j = e_j on sampled columns (any size)
    Ld = L.astype(np.float64)
    for j in np.unique(np.random.default_rng(8).integers(0, n, 4)):
        h = Hrot[:, j].copy()
        h[j] += delta
        r = Ld @ (Ld.T @ h)
        e = np.zeros(n)
        e[j] = 1.0
        assert np.linalg.norm(r - e) <= 1e-3, (j, np.linalg.norm(r - e))


def test_fullsize_sweep_bit_exact(layer):
    cfg, _, p, _, _, Wp = layer
    rows = np.unique(np.random.default_rng(9).integers(0, cfg.d_out, 24))
    Wh = Wp.cpu().numpy()
    Lt32 = np.ascontiguousarray(p.Lt.cpu().numpy())
    c = obs_sweep_fp32(Wh, Lt32, cfg.bits, cfg.group, cfg.block, rows=rows)
    assert np.array_equal(p.codes.cpu().numpy()[rows], c["codes"])
    assert np.array_equal(p.scale.cpu().numpy()[rows], c["scale"])
    assert np.array_equal(p.zero.cpu().numpy()[rows], c["zero"].astype(np.int32))
