"""GPU parity of the GPTAQ drift correction (the full objective, Eq. kronq_full) through the
C ABI, against the oracle on the same seeded inputs:
  * the drift statistic D = (X~ - X)^T X: relative Frobenius error <= 1e-5 against float64,
    and bit-exact where every sum is exact in fp32 (small integers);
  * its rescale and rotation D' = V S_X^-1 D S_X^-1 V^T: <= 1e-5;
  * P = alpha ((D' L) o M_U) L^T, returned as P^T: <= 1e-5 on the GPU's own float32 inputs
    (fp32 arithmetic itself lands near 5e-7 here), exact zeros on and above the diagonal;
  * the sweep with P: bit-exact against the fp32-ordered oracle sweep (fp32 trailing
    update); with the 3xTF32 trailing update the tie rule of the GPTQ-mode sweep;
  * the whole pipeline: the full objective of its codes within 1e-3 of the oracle's, the
    two-stream schedule and the host path giving the same bits as the serialized run.
Stage inputs come from the generator or the oracle, never from another CUDA stage.
"""
import numpy as np
import pytest
import torch

import kqsynth
from oracle import kronq_oracle as ref
from oracle import obs_sweep_fp32

pytestmark = pytest.mark.gpu

DEV = "cuda"
ALPHA = 0.25


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()


def K():
    from paper_2607_07964_gb300 import kronq
    return kronq


def rel_fro(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV).to(dtype)


def bf16_dev(a32):
    return torch.from_numpy(np.ascontiguousarray(a32, dtype=np.float32)).to(DEV).to(torch.bfloat16)


def host(t):
    torch.cuda.synchronize()
    return t.detach().cpu().numpy()


def _drift_inputs(T, d, seed=0):
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=d, d_out=8, T=T, seed=seed, n_outliers=min(4, d))
    X = kqsynth.activations(cfg)
    return cfg, X, kqsynth.fp_activations(cfg, X)


def _gpu_drift(Xt, X, ws_tokens=None, D=None, accumulate=False):
    T, d = X.shape
    if D is None:
        D = torch.full((d, d), float("nan"), device=DEV)
    ws = torch.empty(K().kq_accum_drift_workspace(ws_tokens or max(T, 1), d), dtype=torch.uint8, device=DEV)
    info = torch.zeros(1, dtype=torch.int32, device=DEV)
    K().kq_accum_drift(Xt, X, D, accumulate=accumulate, info=info, ws=ws)
    assert K().kq_check(info)[0] == K().KQ_OK
    return D


# --------------------------------------------------------------------- drift statistic
@pytest.mark.parametrize("T,d", [(4096, 256), (1000, 384), (777, 896), (64, 16), (130, 8), (2048, 1024)])
def test_drift_factor_parity(T, d):
    _, X, Xt = _drift_inputs(T, d, seed=d)
    Dg = host(_gpu_drift(bf16_dev(Xt), bf16_dev(X)))
    Dref = ref.drift_factor(Xt, X)
    assert rel_fro(Dg, Dref) <= 1e-5
    assert not np.allclose(Dg, Dg.T)


def test_drift_factor_exact_on_integers():
    """Small integers: every product and partial sum is exact in fp32, so D is exact."""
    rng = np.random.default_rng(4)
    T, d = 512, 64
    X = rng.integers(-8, 9, size=(T, d)).astype(np.float32)
    Xt = X + rng.integers(-3, 4, size=(T, d)).astype(np.float32)
    Dg = host(_gpu_drift(bf16_dev(Xt), bf16_dev(X)))
    assert np.array_equal(Dg, ref.drift_factor(Xt, X).astype(np.float32))


def test_drift_factor_chunks_accumulate_and_stride():
    """A workspace of 128 tokens (the call runs 8 token chunks), accumulate = 1, and a
    column slice (row stride 2 d) of wider matrices."""
    _, X, Xt = _drift_inputs(1000, 512, seed=3)
    d = 256
    Xd, Xtd = bf16_dev(X), bf16_dev(Xt)
    Dref = ref.drift_factor(Xt[:, :d], X[:, :d])
    D = _gpu_drift(Xtd[:, :d], Xd[:, :d], ws_tokens=128)
    assert rel_fro(host(D), Dref) <= 1e-5
    _gpu_drift(Xtd[:, :d], Xd[:, :d], ws_tokens=128, D=D, accumulate=True)
    assert rel_fro(host(D), 2 * Dref) <= 1e-5


def test_drift_factor_wide_exponent_gaps():
    """Drift values whose two bf16 operands are far apart in exponent (x~ = 300 x, x~ = 0):
    the hi + lo pair no longer holds them exactly, but within 2^-17."""
    _, X, Xt = _drift_inputs(2048, 256, seed=9)
    rng = np.random.default_rng(2)
    Xt = Xt.copy()
    m = rng.random(Xt.shape) < 0.05
    Xt[m] = kqsynth.round_bf16(300.0 * X[m])
    Xt[rng.random(Xt.shape) < 0.05] = 0.0
    Dg = host(_gpu_drift(bf16_dev(Xt), bf16_dev(X)))
    assert rel_fro(Dg, ref.drift_factor(Xt, X)) <= 1e-5


def test_drift_factor_empty():
    D = torch.full((16, 16), 3.0, device=DEV)
    X = torch.zeros((0, 16), dtype=torch.bfloat16, device=DEV)
    ws = torch.empty(256, dtype=torch.uint8, device=DEV)
    K().kq_accum_drift(X, X, D, accumulate=True, ws=ws)
    assert np.all(host(D) == 3.0)
    K().kq_accum_drift(X, X, D, accumulate=False, ws=ws)
    assert np.all(host(D) == 0.0)


@pytest.mark.parametrize("d", [256, 896])
def test_drift_rotation_parity(d):
    """Alg. 1: D' = V S_X^-1 D S_X^-1 V^T through kq_rotate_in (W = NULL)."""
    cfg, X, Xt = _drift_inputs(4 * d, d, seed=d + 1)
    D32 = ref.drift_factor(Xt, X).astype(np.float32)
    s_x = np.exp(np.random.default_rng(d).standard_normal(d) * 0.5).astype(np.float32)
    _, sv = kqsynth.signs(cfg)
    Dd = dev(D32)
    K().kq_rotate_in(None, Dd, dev(s_x), dev(sv, torch.int8), K().KQ_FWD)
    V = ref.rht_matrix(d, sv)
    sx = s_x.astype(np.float64)
    want = V @ (D32.astype(np.float64) / sx[:, None] / sx[None, :]) @ V.T
    assert rel_fro(host(Dd), want) <= 1e-5


# --------------------------------------------------------------------------------- P
def _p_inputs(n, seed):
    """A drift statistic after BiIP and the lower factor of the damped H_X', as float32."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=n, d_out=8, T=4 * n, seed=seed, n_outliers=min(4, n))
    X = kqsynth.activations(cfg)
    Xt = kqsynth.fp_activations(cfg, X)
    H = ref.accum_factor(X)
    Dm = ref.drift_factor(Xt, X)
    sx = np.sqrt(np.sqrt(np.diag(H)))
    Lt = ref.lower_factor(ref.damp(H / sx[:, None] / sx[None, :], 0.01)).astype(np.float32)
    Dp = (Dm / sx[:, None] / sx[None, :]).astype(np.float32)
    return Dp, Lt


def _gpu_p(Dp, Lt, alpha=ALPHA):
    n = Lt.shape[0]
    Pt = torch.full((n, n), float("nan"), device=DEV)
    ws = torch.empty(K().kq_gptaq_p_workspace(n), dtype=torch.uint8, device=DEV)
    info = torch.zeros(1, dtype=torch.int32, device=DEV)
    K().kq_gptaq_p(dev(Dp), dev(Lt), alpha, Pt, ws, info=info)
    assert K().kq_check(info)[0] == K().KQ_OK
    return host(Pt)


@pytest.mark.parametrize("n", [256, 640, 200, 1024, 28 * 32])
def test_gptaq_p_parity(n):
    Dp, Lt = _p_inputs(n, seed=n)
    Pt = _gpu_p(Dp, Lt)
    P = ref.gptaq_p(Dp.astype(np.float64), Lt.astype(np.float64), ALPHA)
    assert np.all(np.triu(Pt) == 0), "P^T is strictly lower triangular"
    assert rel_fro(Pt, P.T) <= 1e-5


def test_gptaq_p_zero_drift_and_linearity():
    Dp, Lt = _p_inputs(384, seed=5)
    assert np.all(_gpu_p(np.zeros_like(Dp), Lt) == 0)
    a = _gpu_p(Dp, Lt, 1.0)
    b = _gpu_p(Dp, Lt, 0.25)
    assert np.array_equal(b, np.float32(0.25) * a)   # alpha scales the last rounding only


# ----------------------------------------------------------------------- the sweep
def _sweep_inputs(d_out, d_in, seed):
    Dp, Lt = _p_inputs(d_in, seed)
    P = ref.gptaq_p(Dp.astype(np.float64), Lt.astype(np.float64), ALPHA)
    Pt = np.ascontiguousarray(P.T).astype(np.float32)
    rng = np.random.default_rng(seed)
    Wp = (rng.standard_normal((d_out, d_in)) * 0.05).astype(np.float32)
    return Wp, Lt, Pt


def _gpu_sweep(Wp, Lt, Pt, bits, group, mode=0):
    d_out, d_in = Wp.shape
    ng = 1 if group == 0 else -(-d_in // group)
    codes = torch.empty((d_out, d_in), dtype=torch.uint8, device=DEV)
    scale = torch.empty((d_out, ng), device=DEV)
    zero = torch.empty((d_out, ng), dtype=torch.int32, device=DEV)
    col_loss = torch.empty(d_in, device=DEV)
    pre_q = torch.empty((d_out, d_in), device=DEV)
    ws = torch.empty(K().kq_obs_quantize_workspace(d_out, d_in, 128, mode, True), dtype=torch.uint8, device=DEV)
    info = torch.zeros(1, dtype=torch.int32, device=DEV)
    K().kq_obs_quantize(dev(Wp), dev(Lt), bits, group, 128, codes, scale, zero, col_loss, pre_q, ws, mode=mode,
                        info=info, Pt=dev(Pt))
    assert K().kq_check(info)[0] == K().KQ_OK
    return {"codes": host(codes), "scale": host(scale), "zero": host(zero), "col_loss": host(col_loss),
            "pre_q": host(pre_q)}


@pytest.mark.parametrize("d_out,d_in,bits,group", [
    (256, 256, 4, 128), (100, 384, 3, 128), (64, 896, 2, 0), (300, 512, 8, 128), (37, 1024, 4, 128),
    (16, 128, 2, 0)])
def test_sweep_with_p_bit_exact(d_out, d_in, bits, group):
    Wp, Lt, Pt = _sweep_inputs(d_out, d_in, seed=d_in + bits)
    g = _gpu_sweep(Wp, Lt, Pt, bits, group)
    c = obs_sweep_fp32(Wp, Lt, bits, group, 128, want_pre_q=True, Pt=Pt)
    assert np.array_equal(g["codes"], c["codes"])
    assert np.array_equal(g["scale"], c["scale"])
    assert np.array_equal(g["zero"], c["zero"].astype(np.int32))
    assert np.array_equal(g["pre_q"], c["pre_q"])
    assert np.allclose(g["col_loss"], np.sum(c["E"].astype(np.float64) ** 2, axis=0), rtol=1e-6, atol=0)
    # the correction is active: GPTQ mode gives other codes
    assert not np.array_equal(c["codes"], obs_sweep_fp32(Wp, Lt, bits, group, 128)["codes"])


@pytest.mark.parametrize("d_out,d_in,bits,group", [
    (256, 256, 4, 128), (300, 1024, 4, 128), (512, 896, 3, 128), (128, 1536, 2, 0), (5120, 1024, 3, 128)])
def test_sweep_with_p_tensor_core_trailing(d_out, d_in, bits, group):
    """3xTF32 trailing update with K = 256 ([E | -Wpre] [R ; P]): teacher forced on every row
    (with the P terms), and the tie rule against the fp32-ordered sweep (<= 0.1 % of codes
    differ, each row's first difference at a rounding tie). (5120, 1024) has more row CTAs
    than SMs."""
    from sweep_checks import check_against_fp32_sweep, check_teacher_forced
    Wp, Lt, Pt = _sweep_inputs(d_out, d_in, seed=d_in + 7 * bits)
    g = _gpu_sweep(Wp, Lt, Pt, bits, group, mode=K().KQ_TRAIL_3XTF32)
    check_teacher_forced(Wp, Lt, g, bits, group, 128, Pt=Pt)
    rows = np.sort(np.random.default_rng(4).choice(d_out, 64, replace=False)) if d_out > 1024 else None
    c, mis = check_against_fp32_sweep(Wp, Lt, g, bits, group, 128, Pt=Pt, rows=rows)
    sel = slice(None) if rows is None else rows
    same = ~mis.any(axis=1)
    ng = c["scale"].shape[1]
    step = np.repeat(c["scale"], 128, axis=1)[:, :d_in] if ng > 1 else c["scale"]
    assert np.max((np.abs(g["pre_q"][sel] - c["pre_q"]) / step)[same]) <= 1e-4


# ------------------------------------------------------------------- whole pipeline
def _layer(d_out, d_in, T, bits, group, seed=0):
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_out=d_out, d_in=d_in, T=T, bits=bits, group=group, seed=seed,
                                             w_bf16=True)
    L = kqsynth.layer(cfg)
    L["Xt"] = kqsynth.fp_activations(cfg, L["X"])
    return cfg, L


def _gpu_pipeline(cfg, L, trailing="fp32", overlap=False, host_path=False):
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, trailing=trailing,
                      overlap=overlap, alpha=ALPHA, g_chunk_tokens=0)
    if host_path:
        pin = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(dt).pin_memory()  # noqa: E731
        codes = torch.empty(p.codes.shape, dtype=torch.uint8).pin_memory()
        scale = torch.empty(p.scale.shape).pin_memory()
        zero = torch.empty(p.zero.shape, dtype=torch.int32).pin_memory()
        p.run_host(pin(L["X"], torch.bfloat16), pin(L["G"], torch.bfloat16), pin(L["W"], torch.float32),
                   pin(L["sign_u"], torch.int8), pin(L["sign_v"], torch.int8), codes, scale, zero,
                   Xt_h=pin(L["Xt"], torch.bfloat16))
        torch.cuda.synchronize()
        p.check()
        return p
    p.run(bf16_dev(L["X"]), bf16_dev(L["G"]), dev(L["W"]), dev(L["sign_u"], torch.int8),
          dev(L["sign_v"], torch.int8), Xt=bf16_dev(L["Xt"]))
    p.check()
    return p


@pytest.mark.parametrize("trailing", ["fp32", "3xtf32"])
def test_pipeline_with_drift_objective(trailing):
    """The full objective of Eq. (kronq_full), evaluated in float64 on the reverted GPU
    weights, within 1e-3 of the oracle pipeline's (same inputs, same alpha)."""
    cfg, L = _layer(256, 512, 4096, 3, 128)
    o = ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], cfg.bits, cfg.group, cfg.block,
                     cfg.damp, Xt=L["Xt"], alpha=ALPHA)
    p = _gpu_pipeline(cfg, L, trailing)
    W = dev(L["W"])
    What = torch.empty_like(W)
    K().kq_dequant_revert(p.codes, p.scale, p.zero, cfg.group, p.s_x, p.s_g, dev(L["sign_u"], torch.int8),
                          dev(L["sign_v"], torch.int8), What)
    HX, HG = ref.accum_factor(L["X"]), ref.accum_factor(L["G"])
    j_gpu = ref.objective(L["W"], host(What), HX, HG, o["D"])
    first = ref.proxy_loss(L["W"], o["What"], HX, HG)
    assert abs(j_gpu - o["objective"]) <= 1e-3 * (first + abs(o["objective"] - first))
    assert np.mean(host(p.codes) == o["codes"]) > 0.97
    # the correction is active: the drift-corrected codes differ from GPTQ mode's
    g = ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], cfg.bits, cfg.group, cfg.block, cfg.damp)
    assert np.mean(g["codes"] != o["codes"]) > 0.01


def test_pipeline_with_drift_schedules_agree():
    """Serialized, two-stream and host-path runs of the drift pipeline give the same bits
    (fp32-ordered trailing update: every result is deterministic)."""
    cfg, L = _layer(224, 896, 3000, 4, 128, seed=2)
    a = _gpu_pipeline(cfg, L, overlap=False)
    b = _gpu_pipeline(cfg, L, overlap=True)
    c = _gpu_pipeline(cfg, L, overlap=True, host_path=True)
    for q in (b, c):
        assert np.array_equal(host(a.codes), host(q.codes))
        assert np.array_equal(host(a.scale), host(q.scale))
        assert np.array_equal(host(a.Pt), host(q.Pt))
