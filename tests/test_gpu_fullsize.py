"""GPU parity at full size for every Llama-shaped layer of the benchmark plan (q_proj and
the MLP layers of the 8B model; q/o, k/v and down_proj of the 70B model), each run the way
the benchmark times it: LayerPipeline.run with the 3xTF32 trailing update, the symmetric
two-sided rotation of H_X (KQ_FWD_SYM), the two-stream schedule and one H_X / H_G launch,
then the same layer as one CUDA graph replay, which must give the same bits. The oracle
cannot redo these layers in float64, so it checks what it can compute one by one, or what
holds at any size:
  * sampled entries and sampled diagonal entries of H_X and H_G (float64 dot products over
    all T tokens), and S_X, S_G at the sampled channels;
  * sampled entries of W' = U S_G W S_X V^T and of H_X' = V S_X^-1 H_X S_X^-1 V^T (rows of
    U and V built one at a time from the Hadamard definition);
  * the whole inverse Cholesky factor against the float64 factor of the damped H_X' the
    GPU produced (relative Frobenius error <= 1e-5), at every size;
  * the sweep on sampled rows: teacher forced (codes = quant(pre_q) bit for bit, pre_q
    within float32 rounding of Algorithm 2 from the GPU's own errors, group grids from the
    block-start values) and against the fp32-ordered oracle (<= 0.1 % of codes differ, the
    first difference in a row at a rounding tie); then the fp32-ordered trailing update
    (the second mode) on the same W' and L, bit-exact on sampled rows.
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
SNAP = ("codes", "scale", "zero", "Lt", "HX", "HG", "s_x", "s_g", "traces", "col_loss", "pre_q", "Wp_in")


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
    args = (inp["X"], inp["G"], inp["W"], inp["sign_u"], inp["sign_v"])
    # the benchmark's pipeline: 3xTF32 sweep, two streams, one H_X and one H_G launch
    p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, trailing="3xtf32",
                      x_chunk_tokens=0, g_chunk_tokens=0, debug_outputs=True)
    p.run(*args)
    p.check()
    snap = {k: getattr(p, k).clone() for k in SNAP}
    graph, _ = p.capture(*args)
    graph.replay()
    torch.cuda.synchronize()
    p.check()
    replay_equal = {k: bool(torch.equal(getattr(p, k), snap[k])) for k in SNAP}
    del graph
    # the raw factors, by the same launches the pipeline makes before it rotates them in place
    HX_raw = torch.empty((cfg.d_in, cfg.d_in), device="cuda")
    HG_raw = torch.empty((cfg.d_out, cfg.d_out), device="cuda")
    K.kq_accum_factor(inp["X"], HX_raw)
    K.kq_accum_factor(inp["G"], HG_raw)
    # the second trailing-update mode (fp32-ordered, bit-exact) on the same W' and L
    ng = snap["scale"].shape[1]
    f32 = {"codes": torch.empty_like(snap["codes"]), "scale": torch.empty_like(snap["scale"]),
           "zero": torch.empty_like(snap["zero"])}
    ws = torch.empty(K.kq_obs_quantize_workspace(cfg.d_out, cfg.d_in, cfg.block, K.KQ_TRAIL_FP32),
                     dtype=torch.uint8, device="cuda")
    info = torch.zeros(1, dtype=torch.int32, device="cuda")
    K.kq_obs_quantize(snap["Wp_in"].clone(), snap["Lt"], cfg.bits, cfg.group, cfg.block, f32["codes"],
                      f32["scale"], f32["zero"], None, None, ws, mode=K.KQ_TRAIL_FP32, info=info)
    assert K.kq_check(info)[0] == K.KQ_OK
    del ws
    assert ng == f32["scale"].shape[1]
    yield cfg, inp, snap, HX_raw, HG_raw, replay_equal, f32
    del p, inp, snap, HX_raw, HG_raw, f32
    torch.cuda.empty_cache()


def test_fullsize_graph_replay_is_bit_identical(layer):
    _, _, _, _, _, replay_equal, _ = layer
    assert all(replay_equal.values()), [k for k, v in replay_equal.items() if not v]


def test_fullsize_factors_and_scales(layer):
    cfg, inp, snap, HX, HG, _, _ = layer
    rng = np.random.default_rng(5)
    W = inp["W"].cpu().numpy().astype(np.float64)
    for A, H, d, s_dev, axis in ((inp["X"], HX, cfg.d_in, snap["s_x"], 0), (inp["G"], HG, cfg.d_out, snap["s_g"], 1)):
        cols = np.unique(rng.integers(0, d, 40))
        Ac = _bf16_cols(A, cols)
        want = Ac.T @ Ac                              # float64 sums over all tokens
        got = H[torch.as_tensor(cols, device="cuda")][:, torch.as_tensor(cols, device="cuda")].cpu().numpy()
        assert _rel(got, want) <= 1e-5
        assert np.max(np.abs(np.diag(got) / np.diag(want) - 1)) <= 1e-5
        # the pipeline's scales at these channels: (h / ||W column or row||^2)^(1/4)
        norm2 = np.sum(W[:, cols] ** 2, axis=0) if axis == 0 else np.sum(W[cols] ** 2, axis=1)
        s_want = (np.diag(want) / norm2) ** 0.25
        assert np.max(np.abs(s_dev.cpu().numpy()[cols] / s_want - 1)) <= 1e-5


def test_fullsize_rotations(layer):
    cfg, inp, snap, HX, HG, _, _ = layer
    rng = np.random.default_rng(6)
    d_out, d_in = cfg.d_out, cfg.d_in
    sx = snap["s_x"].cpu().numpy().astype(np.float64)
    sg = snap["s_g"].cpu().numpy().astype(np.float64)
    su, sv = inp["sign_u"].cpu().numpy(), inp["sign_v"].cpu().numpy()
    rows = np.unique(rng.integers(0, d_out, 12))
    cols = np.unique(rng.integers(0, d_in, 12))
    U = ref.rht_rows(d_out, su, rows)
    V = ref.rht_rows(d_in, sv, cols)
    W = inp["W"].cpu().numpy().astype(np.float64)
    want = ((U * sg[None, :]) @ W * sx[None, :]) @ V.T
    got = snap["Wp_in"].cpu().numpy()[np.ix_(rows, cols)]
    assert _rel(got, want) <= 1e-5
    # H_X' = V S_X^-1 H_X S_X^-1 V^T and H_G' = U S_G^-1 H_G S_G^-1 U^T at sampled entries
    for H, Hp, d, s, sign in ((HX, snap["HX"], d_in, sx, sv), (HG, snap["HG"], d_out, sg, su)):
        a = np.unique(rng.integers(0, d, 10))
        b = np.unique(rng.integers(0, d, 10))
        Hh = H.cpu().numpy().astype(np.float64)
        Va = ref.rht_rows(d, sign, a) / s[None, :]
        Vb = ref.rht_rows(d, sign, b) / s[None, :]
        want = (Va @ Hh) @ Vb.T
        got = Hp.cpu().numpy()[np.ix_(a, b)]
        assert _rel(got, want) <= 1e-5
        del Hh


def test_fullsize_inverse_cholesky(layer):
    """The whole factor against float64: L L^T = (H_X' + lambda mean(diag) I)^-1 with the
    GPU's own H_X' (reverse-order LAPACK route, pinned to the textbook route on the CPU)."""
    cfg, _, snap, _, _, _, _ = layer
    # the matrix as the kernels read it: its upper triangle (the lower one of the reversed
    # matrix), which is also the triangle LAPACK's lower factorization of J H J reads
    Hrot = snap["HX"].cpu().numpy().astype(np.float64)
    Lref = ref.lower_factor_reversed(ref.damp(Hrot, cfg.damp))
    del Hrot
    L = snap["Lt"].cpu().numpy()
    assert np.all(np.triu(L, 1) == 0)
    assert _rel(L, Lref) <= 1e-5


def _sample_rows(d_out, k, seed):
    return np.sort(np.random.default_rng(seed).choice(d_out, min(k, d_out), replace=False))


def test_fullsize_sweep_tensor_core(layer):
    from sweep_checks import check_against_fp32_sweep, check_teacher_forced
    cfg, _, snap, _, _, _, _ = layer
    g = {k: snap[k].cpu().numpy() for k in ("codes", "scale", "zero", "pre_q")}
    Wp = snap["Wp_in"].cpu().numpy()
    Lt = np.ascontiguousarray(snap["Lt"].cpu().numpy())
    check_teacher_forced(Wp, Lt, g, cfg.bits, cfg.group, cfg.block, rows=_sample_rows(cfg.d_out, 64, 9))
    check_against_fp32_sweep(Wp, Lt, g, cfg.bits, cfg.group, cfg.block, rows=_sample_rows(cfg.d_out, 64, 10))


def test_fullsize_sweep_fp32_mode_bit_exact(layer):
    cfg, _, snap, _, _, _, f32 = layer
    rows = _sample_rows(cfg.d_out, 24, 11)
    Wp = snap["Wp_in"].cpu().numpy()
    Lt = np.ascontiguousarray(snap["Lt"].cpu().numpy())
    c = obs_sweep_fp32(Wp, Lt, cfg.bits, cfg.group, cfg.block, rows=rows)
    assert np.array_equal(f32["codes"].cpu().numpy()[rows], c["codes"])
    assert np.array_equal(f32["scale"].cpu().numpy()[rows], c["scale"])
    assert np.array_equal(f32["zero"].cpu().numpy()[rows], c["zero"].astype(np.int32))
