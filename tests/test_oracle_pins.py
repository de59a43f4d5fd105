"""Pins of the float64 oracle against facts the paper and mathematics fix.

None of these compares the oracle with itself: each check is a brute-force sum, a
closed form, an identity from the paper (Theorem 1, Proposition 1, Proposition 2's
equality case, the LDL identity of Proposition 2's proof), a hand-derived worked example
or a special case that reduces to plain rounding.
"""
import json
import os

import numpy as np
import pytest

import kqsynth
from oracle import kronq_oracle as ref
from oracle import obs_sweep_fp32

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- Kronecker factors
def test_factor_brute_force_integers():
    """H = sum_t x_t x_t^T (Eq. ptq_obj with tokens as rows), by Python integer loops."""
    rng = _rng(1)
    T, d = 37, 6
    A = rng.integers(-9, 10, size=(T, d))
    H = ref.accum_factor(A.astype(np.float64))
    brute = [[0] * d for _ in range(d)]
    for t in range(T):
        for i in range(d):
            for j in range(d):
                brute[i][j] += int(A[t, i]) * int(A[t, j])
    assert np.array_equal(H, np.array(brute, dtype=np.float64))


def test_factor_bf16_exact_and_trace():
    """bf16 products are exact in fp64; tr(A^T A) = ||A||_F^2 summed entry by entry."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=16, d_out=8, T=64)
    X = kqsynth.activations(cfg).astype(np.float64)
    H = ref.accum_factor(X)
    tr = 0.0
    for v in X.ravel():
        tr += float(v) * float(v)
    assert np.isclose(np.trace(H), tr, rtol=1e-14)
    # additivity over token chunks (streamed accumulation)
    parts = sum(ref.accum_factor(X[t:t + 16]) for t in range(0, 64, 16))
    assert np.allclose(parts, H, rtol=1e-14, atol=0)


# ---------------------------------------------------------------- Hadamard / RHT
@pytest.mark.parametrize("n", [1, 2, 4, 8, 64, 256, 28, 56, 112, 896])
def test_hadamard_orthogonal_symmetric(n):
    H = ref.hadamard_matrix(n)
    assert set(np.unique(H)) <= {-1, 1}
    assert np.array_equal(H @ H.T, n * np.eye(n, dtype=np.int64))
    assert np.array_equal(H, H.T)


def test_sylvester_h2_and_recursion():
    assert np.array_equal(ref.sylvester(2), np.array([[1, 1], [1, -1]]))
    h4 = ref.sylvester(4)
    for i in range(4):
        for j in range(4):  # entry (i, j) of H_{2^k} is (-1)^{popcount(i & j)}
            assert h4[i, j] == (-1) ** bin(i & j).count("1")


def test_paley28_structure():
    H = ref.paley28()
    assert H.shape == (28, 28)
    assert np.array_equal(H @ H.T, 28 * np.eye(28, dtype=np.int64))
    # expanding the conference matrix's zero diagonal gives the block [[1,-1],[-1,-1]]
    for i in range(14):
        assert np.array_equal(H[2 * i:2 * i + 2, 2 * i:2 * i + 2], [[1, -1], [-1, -1]])


def test_kron_index_layout():
    """n = 28 * 2^k uses index a * 2^k + b: entry = H28[a, a'] * H_{2^k}[b, b']."""
    H = ref.hadamard_matrix(28 * 4)
    h28, h4 = ref.paley28(), ref.sylvester(4)
    for (a, b, a2, b2) in [(0, 0, 0, 0), (3, 1, 5, 2), (27, 3, 1, 3), (13, 2, 13, 1)]:
        assert H[a * 4 + b, a2 * 4 + b2] == h28[a, a2] * h4[b, b2]


@pytest.mark.parametrize("n", [64, 112])
def test_rht_rotate_unrotate(n):
    rng = _rng(n)
    sign = np.where(rng.random(n) < 0.5, -1, 1)
    V = ref.rht_matrix(n, sign)
    assert np.allclose(V @ V.T, np.eye(n), atol=1e-13)
    W = rng.standard_normal((5, n))
    assert np.allclose((W @ V.T) @ V, W, atol=1e-13)
    assert np.allclose(np.linalg.norm(W @ V.T, axis=1), np.linalg.norm(W, axis=1))


@pytest.mark.parametrize("n", [8, 64, 28, 112, 896])
def test_rht_rows_match_dense_matrix(n):
    """The row-at-a-time RHT used at full size equals rows of the dense definition."""
    rng = _rng(n + 1)
    sign = np.where(rng.random(n) < 0.5, -1, 1)
    rows = np.unique(rng.integers(0, n, 5))
    assert np.array_equal(ref.rht_rows(n, sign, rows), ref.rht_matrix(n, sign)[rows])


def test_rht_rows_orthonormal_at_large_size():
    """Rows of V for n = 28 * 1024 are orthonormal (checked on a sample)."""
    n = 28 * 1024
    sign = np.where(_rng(3).random(n) < 0.5, -1, 1)
    R = ref.rht_rows(n, sign, [0, 1, 1023, 1024, 20000, n - 1])
    assert np.allclose(R @ R.T, np.eye(6), atol=1e-12)


# ---------------------------------------------------------------- rescaling (Eq. rescale)
def test_rescale_equalizes_norms_and_diagonals():
    """With S_X = (h/a)^(1/4), the rescaled column energy a_j s_j^2 equals the rescaled
    Hessian diagonal h_j / s_j^2 (= sqrt(h_j a_j)); any other exponent breaks this."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=32, d_out=24, T=256)
    L = kqsynth.layer(cfg)
    HX, HG = ref.accum_factor(L["X"]), ref.accum_factor(L["G"])
    W = L["W"].astype(np.float64)
    sx, sg = ref.biip_scales(W, HX, HG)
    a, r = np.sum(W * W, 0), np.sum(W * W, 1)
    assert np.allclose(a * sx ** 2, np.diag(HX) / sx ** 2, rtol=1e-12)
    assert np.allclose(r * sg ** 2, np.diag(HG) / sg ** 2, rtol=1e-12)
    assert np.allclose(a * sx ** 2, np.sqrt(np.diag(HX) * a), rtol=1e-12)


def test_prop2_cauchy_schwarz_equality():
    """Prop. 2: (sum h/s^2)(sum s^2 a) >= (sum sqrt(h a))^2 with equality at the S_G of
    Eq. (rescale); the gain rho = (sum sqrt(h a))^2 / (sum h sum a) <= 1."""
    rng = _rng(7)
    h = np.exp(3 * rng.standard_normal(50))
    W = rng.standard_normal((50, 40))
    a = np.sum(W * W, 1)
    HG = np.diag(h)
    _, s = ref.biip_scales(W, np.eye(40), HG)
    lhs = np.sum(h / s ** 2) * np.sum(s ** 2 * a)
    assert np.isclose(lhs, np.sum(np.sqrt(h * a)) ** 2, rtol=1e-12)
    s_half = (h / a) ** 0.5
    assert np.sum(h / s_half ** 2) * np.sum(s_half ** 2 * a) > lhs * (1 + 1e-3)
    rho = np.sum(np.sqrt(h * a)) ** 2 / (np.sum(h) * np.sum(a))
    assert 0 < rho < 1


def test_dead_channel_scale_is_one():
    W = np.ones((4, 3))
    W[:, 1] = 0.0
    HX = np.diag([4.0, 2.0, 0.0])
    sx, _ = ref.biip_scales(W, HX, np.eye(4))
    assert sx[1] == 1.0 and sx[2] == 1.0 and np.isclose(sx[0], (4.0 / 4.0) ** 0.25)


# ---------------------------------------------------------------- Theorem 1
def test_theorem1_objective_invariance():
    """tr(H_G dW H_X dW^T) is the same in the original and the BiIP space for any W^."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=56, d_out=32, T=512)
    L = kqsynth.layer(cfg)
    HX, HG = ref.accum_factor(L["X"]), ref.accum_factor(L["G"])
    W = L["W"].astype(np.float64)
    b = ref.biip(W, HX, HG, L["sign_u"], L["sign_v"])
    rng = _rng(3)
    Qp = b["W"] + 0.01 * rng.standard_normal(b["W"].shape)
    What = ref.revert(Qp, b["s_x"], b["s_g"], b["U"], b["V"])
    l_orig = ref.proxy_loss(W, What, HX, HG)
    l_rot = ref.proxy_loss(b["W"], Qp, b["HX"], b["HG"])
    assert np.isclose(l_orig, l_rot, rtol=1e-9)
    # reverting the unquantized W' gives back W exactly
    assert np.allclose(ref.revert(b["W"], b["s_x"], b["s_g"], b["U"], b["V"]), W, atol=1e-12)


def test_proxy_loss_is_kronecker_quadratic():
    """Eq. (kfac)/(kron_obj): vec(dW)^T (H_X kron H_G) vec(dW), vec stacking columns."""
    rng = _rng(11)
    m, n = 4, 5
    A, B = rng.standard_normal((9, n)), rng.standard_normal((9, m))
    HX, HG = A.T @ A, B.T @ B
    W, What = rng.standard_normal((m, n)), rng.standard_normal((m, n))
    v = (W - What).reshape(-1, order="F")
    assert np.isclose(ref.proxy_loss(W, What, HX, HG), v @ np.kron(HX, HG) @ v, rtol=1e-12)


def test_post_biip_traces():
    """RHTs preserve the trace: tr(V S^-1 H S^-1 V^T) = sum_j h_j / s_j^2 = sum sqrt(h a)."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=64, d_out=28, T=300)
    L = kqsynth.layer(cfg)
    out = ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], 4, 0, 32)
    W = L["W"].astype(np.float64)
    a, r = np.sum(W * W, 0), np.sum(W * W, 1)
    assert np.isclose(out["trHX_post"], np.sum(np.sqrt(np.diag(out["HX"]) * a)), rtol=1e-12)
    assert np.isclose(out["trHG_post"], np.sum(np.sqrt(np.diag(out["HG"]) * r)), rtol=1e-12)
    assert np.isclose(out["trHX"], np.sum(L["X"].astype(np.float64) ** 2), rtol=1e-12)
    assert np.isclose(out["s_post"], out["trHX_post"] * out["trHG_post"])


# ---------------------------------------------------------------- inverse Cholesky
def _textbook_reverse_route(H):
    """Pure-Python route independent of the library one: factor H = U U^T with U upper
    (Cholesky from the bottom-right corner), then R = U^-1 by back substitution."""
    n = len(H)
    U = [[0.0] * n for _ in range(n)]
    A = [list(map(float, row)) for row in H]
    for k in range(n - 1, -1, -1):
        U[k][k] = A[k][k] ** 0.5
        for i in range(k):
            U[i][k] = A[i][k] / U[k][k]
        for i in range(k):
            for j in range(k):
                A[i][j] -= U[i][k] * U[j][k]
    R = [[0.0] * n for _ in range(n)]
    for j in range(n):           # solve U R = I column by column (R upper)
        for i in range(j, -1, -1):
            s = 1.0 if i == j else 0.0
            for k in range(i + 1, j + 1):
                s -= U[i][k] * R[k][j]
            R[i][j] = s / U[i][i]
    return np.array(R)


def test_inverse_cholesky_routes_agree():
    H = ref.damp(kqsynth.random_spd(12, seed=5), 0.01)
    R = ref.inverse_cholesky_upper(H)
    assert np.allclose(np.triu(R), R) and np.all(np.diag(R) > 0)
    assert np.allclose(R.T @ R @ H, np.eye(12), atol=1e-9)
    assert np.allclose(_textbook_reverse_route(H), R, rtol=1e-9, atol=1e-12)
    assert np.array_equal(ref.lower_factor(H), R.T)


@pytest.mark.parametrize("n", [12, 300])
def test_inverse_cholesky_reversed_route_is_the_textbook_factor(n):
    """The LAPACK reverse-order route used for the largest layers' checks gives the textbook
    factor (the lower Cholesky-type factor of H^-1 with a positive diagonal is unique)."""
    H = ref.damp(kqsynth.random_spd(n, seed=n), 0.01)
    L = ref.lower_factor(H)
    Lr = ref.lower_factor_reversed(H)
    assert np.array_equal(np.triu(Lr, 1), np.zeros_like(Lr)) and np.all(np.diag(Lr) > 0)
    assert np.allclose(Lr, L, rtol=1e-9, atol=1e-12 * np.abs(L).max())
    assert np.allclose(Lr @ Lr.T @ H, np.eye(n), atol=1e-8)


def test_obs_row_is_inverse_of_remaining_block():
    """Eq. (obs_update): R[p, p:]/R[p, p] = [H_F^-1]_{p, :}/[H_F^-1]_{pp}, F = {p, .., n-1}."""
    H = ref.damp(kqsynth.random_spd(10, seed=9), 0.01)
    R = ref.inverse_cholesky_upper(H)
    for p in range(10):
        HFi = np.linalg.inv(H[p:, p:])
        assert np.allclose(R[p, p:] / R[p, p], HFi[0] / HFi[0, 0], rtol=1e-9, atol=1e-12)
        assert np.isclose(R[p, p] ** 2, HFi[0, 0], rtol=1e-10)


def test_damping_is_relative_to_mean_diagonal():
    H = np.diag([1.0, 3.0])
    assert np.allclose(ref.damp(H, 0.5), np.diag([2.0, 4.0]))


# ---------------------------------------------------------------- quantizer
def test_quantizer_grid_points_and_ties():
    s, z = ref.quant_params(np.array([[-1.0, 0.5, 2.0]]), 2)  # scale = 3/3 = 1, zero = 1
    assert s[0] == 1.0 and z[0] == 1.0
    grid = s[0] * (np.arange(4) - z[0])
    assert np.array_equal(ref.quantize(grid, s[0], z[0], 2), np.arange(4))
    # ties to even: 0.5 -> 0, 1.5 -> 2, -0.5 -> -0; plus zero
    assert np.array_equal(ref.quantize(np.array([0.5, 1.5, -0.5]), 1.0, 1.0, 2), [1, 3, 1])
    # clamping and the all-zero row
    assert ref.quantize(np.array([100.0]), 1.0, 1.0, 2)[0] == 3
    s0, z0 = ref.quant_params(np.zeros((1, 4)), 3)
    assert s0[0] == 2.0 / 7 and z0[0] == np.rint(7 / 2)
    # min-max grid: dequantized error at most scale/2 inside the range
    x = _rng(2).standard_normal((3, 50))
    s, z = ref.quant_params(x, 4)
    q = ref.quantize(x, s[:, None], z[:, None], 4)
    assert np.all(np.abs(s[:, None] * (q - z[:, None]) - x) <= s[:, None] / 2 + 1e-12)


# ---------------------------------------------------------------- OBS sweep
def test_worked_example_golden():
    g = json.load(open(os.path.join(GOLDEN, "obs_worked_2col.json")))
    R = ref.inverse_cholesky_upper(np.array(g["H"]))
    assert np.allclose(R, g["R"], rtol=1e-14)
    sw = ref.obs_sweep(np.array(g["W"]), R, g["bits"], 0, 128)
    assert sw["codes"].tolist() == g["codes"]
    assert np.isclose(sw["scale"][0, 0], g["scale"]) and sw["zero"][0, 0] == g["zero"]
    assert np.allclose(sw["pre_q"], g["pre_q"], rtol=1e-14)
    assert np.allclose(sw["E"], g["E"], rtol=1e-13)
    assert np.isclose(np.sum(sw["E"] ** 2), g["loss"], rtol=1e-13)
    # the fp32-ordered C sweep gives the same codes on the same example
    c = obs_sweep_fp32(np.array(g["W"], np.float32), R.T.astype(np.float32), g["bits"], 0, 128)
    assert c["codes"].tolist() == g["codes"]


@pytest.mark.parametrize("group,block", [(0, 16), (16, 16), (0, 128)])
def test_identity_hessian_reduces_to_rtn(group, block):
    """H = c I (R diagonal): no compensation, the sweep is round-to-nearest on the grid."""
    rng = _rng(4)
    W = rng.standard_normal((20, 48)) * 0.02
    R = ref.inverse_cholesky_upper(2.5 * np.eye(48))
    sw = ref.obs_sweep(W, R, 3, group, block)
    if group == 0:
        s, z = ref.quant_params(W, 3)
        rtn = np.clip(np.rint(W / s[:, None]) + z[:, None], 0, 7)
    else:
        rtn = np.zeros_like(W)
        for g0 in range(0, 48, group):
            s, z = ref.quant_params(W[:, g0:g0 + group], 3)
            rtn[:, g0:g0 + group] = np.clip(np.rint(W[:, g0:g0 + group] / s[:, None]) + z[:, None], 0, 7)
    assert np.array_equal(sw["codes"], rtn.astype(np.uint8))
    assert np.array_equal(sw["pre_q"], W)
    c = obs_sweep_fp32(W.astype(np.float32), R.T.astype(np.float32), 3, group, block)
    W32 = W.astype(np.float32)
    if group == 0:
        s32 = c["scale"][:, 0]
        z32 = c["zero"][:, 0]
        rtn32 = np.clip(np.rint(W32 / s32[:, None]) + z32[:, None], 0, 7)
        assert np.array_equal(c["codes"], rtn32.astype(np.uint8))


@pytest.mark.parametrize("group,block", [(0, 8), (8, 8), (0, 32)])
def test_ldl_identity(group, block):
    """Proof of Prop. 2 (e H e^T = eta D eta^T): sum_j sum_rows E_j^2 = tr(dW H dW^T)."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=32, d_out=16, T=200)
    L = kqsynth.layer(cfg)
    H = ref.damp(ref.accum_factor(L["X"]), 0.01)
    R = ref.inverse_cholesky_upper(H)
    W = L["W"].astype(np.float64)
    sw = ref.obs_sweep(W, R, 2, group, block)
    dW = W - ref.dequant(sw["codes"], sw["scale"], sw["zero"], group)
    assert np.isclose(np.sum(sw["E"] ** 2), np.trace(dW @ H @ dW.T), rtol=1e-10)


@pytest.mark.parametrize("block", [4, 32])
def test_sequential_least_squares(block):
    """Each compensated column equals the fp64 argmin of the quadratic with the earlier
    columns fixed at their quantized values: w_F + (w_Q - q_Q) H_QF H_FF^-1."""
    n = 20
    H = ref.damp(kqsynth.random_spd(n, seed=13), 0.01)
    R = ref.inverse_cholesky_upper(H)
    W = _rng(5).standard_normal((6, n)) * 0.05
    sw = ref.obs_sweep(W, R, 3, 0, block)
    Q = ref.dequant(sw["codes"], sw["scale"], sw["zero"], 0)
    for p in range(1, n):
        Qi, F = slice(0, p), slice(p, n)
        comp = W[:, F] + (W[:, Qi] - Q[:, Qi]) @ H[Qi, F] @ np.linalg.inv(H[F, F])
        assert np.allclose(sw["pre_q"][:, p], comp[:, 0], rtol=1e-9, atol=1e-12)


def test_prop1_hg_offdiagonal_does_not_change_codes():
    """Prop. 1: H_G cancels in the update; only diag(H_G) reaches the sweep (through S_G)."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=32, d_out=28, T=400)
    L = kqsynth.layer(cfg)
    a = ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], 3, 0, 16)
    HG = ref.accum_factor(L["G"])
    HG2 = np.diag(np.diag(HG)) + 0.3 * (HG - np.diag(np.diag(HG)))
    HX = ref.accum_factor(L["X"])
    b = ref.biip(L["W"], HX, HG2, L["sign_u"], L["sign_v"])
    sw = ref.obs_sweep(b["W"], ref.inverse_cholesky_upper(ref.damp(b["HX"], 0.01)), 3, 0, 16)
    assert np.array_equal(sw["codes"], a["codes"])


def test_greedy_sweep_bounded_by_brute_force():
    """Tiny layers: the sweep is greedy, so its loss (which equals the quadratic of its
    own codes) is bounded below by the optimum over all grid codes (brute force)."""
    rng = _rng(21)
    for trial in range(5):
        n = 4
        H = ref.damp(kqsynth.random_spd(n, seed=30 + trial), 0.01)
        R = ref.inverse_cholesky_upper(H)
        w = rng.standard_normal((1, n))
        sw = ref.obs_sweep(w, R, 2, 0, 128)
        s, z = sw["scale"][0, 0], sw["zero"][0, 0]
        loss = np.sum(sw["E"] ** 2)
        best = np.inf
        for code in np.ndindex(*(4,) * n):
            d = w[0] - s * (np.array(code) - z)
            best = min(best, d @ H @ d)
        d = w[0] - s * (sw["codes"][0] - z)
        assert np.isclose(loss, d @ H @ d, rtol=1e-10)
        assert best - 1e-12 <= loss


# ---------------------------------------------------------------- fp32-ordered C sweep
@pytest.mark.parametrize("group", [0, 32])
def test_fp32_sweep_matches_fp64_off_ties(group):
    """The fp32-ordered sweep agrees with the fp64 sweep wherever the decision is not
    within fp32 noise of a rounding tie, and its losses agree to fp32 accuracy."""
    n, m = 64, 40
    H = ref.damp(kqsynth.random_spd(n, seed=17), 0.01)
    R = ref.inverse_cholesky_upper(H)
    R32 = R.astype(np.float32)
    W32 = (_rng(8).standard_normal((m, n)) * 0.02).astype(np.float32)
    s64 = ref.obs_sweep(W32.astype(np.float64), R32.astype(np.float64), 4, group, 32)
    s32 = obs_sweep_fp32(W32, R32.T, 4, group, 32)
    diff = s64["codes"] != s32["codes"]
    # rows diverge after a flipped decision; the first flip in each row must be a near-tie
    for r in np.nonzero(diff.any(1))[0]:
        j = np.argmax(diff[r])
        g = 0 if group == 0 else j // group
        t = s64["pre_q"][r, j] / s64["scale"][r, g]
        assert abs(abs(t - np.floor(t)) - 0.5) < 1e-3
    assert diff.mean() < 0.02
    assert np.isclose(np.sum(s32["E"].astype(np.float64) ** 2), np.sum(s64["E"] ** 2), rtol=1e-3)


def test_fp32_sweep_row_subset():
    n, m = 48, 12
    H = ref.damp(kqsynth.random_spd(n, seed=3), 0.01)
    Lt = ref.lower_factor(H).astype(np.float32)
    W = (_rng(9).standard_normal((m, n)) * 0.02).astype(np.float32)
    full = obs_sweep_fp32(W, Lt, 3, 16, 16)
    rows = np.array([7, 0, 11])
    part = obs_sweep_fp32(W, Lt, 3, 16, 16, rows=rows)
    assert np.array_equal(part["codes"], full["codes"][rows])
    assert np.array_equal(part["E"], full["E"][rows])


# ------------------------------------------------------------- teacher-forced replay
def _tf_problem(n=96, m=30, seed=21, with_p=False):
    H = ref.damp(kqsynth.random_spd(n, seed=seed), 0.01)
    Lt = ref.lower_factor(H).astype(np.float32)
    W = (_rng(seed + 1).standard_normal((m, n)) * 0.02).astype(np.float32)
    Pt = None
    if with_p:
        X, Xt, _, _, _, _ = _drift_problem(seed + 2, T=4 * n, n=n)
        P = ref.gptaq_p(ref.drift_factor(Xt, X), Lt.astype(np.float64), 0.25)
        Pt = np.ascontiguousarray(P.T.astype(np.float32))
    return W, Lt, Pt


@pytest.mark.parametrize("group,with_p", [(0, False), (32, False), (32, True)])
def test_teacher_forced_replays_the_fp32_sweep(group, with_p):
    """Fed the fp32-ordered sweep's own decisions, the replay returns that sweep's errors
    bit for bit and its codes exactly, puts its pre-quantization values within float32
    rounding of the exact compensation, and draws its group grids from the block-start
    values."""
    W, Lt, Pt = _tf_problem(with_p=with_p)
    c = obs_sweep_fp32(W, Lt, 3, group, 32, want_pre_q=True, Pt=Pt)
    tf = ref.teacher_forced(W, Lt, c["pre_q"], c["codes"], c["scale"], c["zero"], 3, group, 32, Pt=Pt)
    assert np.array_equal(tf["E"], c["E"])
    assert np.array_equal(tf["codes"], c["codes"])
    dev = np.abs(tf["pre_q"] - c["pre_q"]) / tf["absum"]
    assert dev.max() <= 2e-6, dev.max()
    if group:
        for g in range(W.shape[1] // group):
            s, _ = ref.quant_params(tf["block_start"][:, g * group:(g + 1) * group], 3)
            assert np.allclose(s, c["scale"][:, g], rtol=1e-5, atol=0)
    else:
        assert "block_start" not in tf


def test_teacher_forced_catches_planted_errors():
    """Sweeps with a planted mistake fail the replay: one block's lazy update dropped, the
    compensation's sign flipped, one code off by one."""
    W, Lt, _ = _tf_problem()
    group, block = 32, 32
    good = obs_sweep_fp32(W, Lt, 3, group, block, want_pre_q=True)

    def worst(run):
        tf = ref.teacher_forced(W, Lt, run["pre_q"], run["codes"], run["scale"], run["zero"], 3, group, block)
        return float(np.max(np.abs(tf["pre_q"] - run["pre_q"]) / tf["absum"])), tf

    assert worst(good)[0] <= 2e-6
    dropped = Lt.copy()
    dropped[64:, 32:64] = 0.0          # R[32:64, 64:] = 0: block 1 never updates the later blocks
    assert worst(obs_sweep_fp32(W, dropped, 3, group, block, want_pre_q=True))[0] > 1e-3
    flipped = Lt.copy()
    off = np.tril(np.ones_like(Lt, dtype=bool), -1)
    flipped[off] = -flipped[off]       # every compensation with the wrong sign
    assert worst(obs_sweep_fp32(W, flipped, 3, group, block, want_pre_q=True))[0] > 1e-3
    codes = good["codes"].copy()
    codes[3, 40] = codes[3, 40] + 1 if codes[3, 40] < 7 else codes[3, 40] - 1
    _, tf = worst(dict(good, codes=codes))
    assert not np.array_equal(tf["codes"], codes)


def test_gpu_sweep_checks_accept_the_definition_and_reject_a_planted_error():
    """The fast-mode checks the GPU tests apply (tests/sweep_checks.py) pass on the
    fp32-ordered sweep itself and fail on a sweep that drops one block's lazy update."""
    from sweep_checks import check_fast_sweep
    W, Lt, _ = _tf_problem(n=256, m=40)
    good = obs_sweep_fp32(W, Lt, 3, 128, 128, want_pre_q=True)
    check_fast_sweep(W, Lt, good, 3, 128, 128)
    dropped = Lt.copy()
    dropped[128:, :128] *= np.float32(0.5)    # half of block 0's update of block 1
    bad = obs_sweep_fp32(W, dropped, 3, 128, 128, want_pre_q=True)
    with pytest.raises(AssertionError):
        check_fast_sweep(W, Lt, bad, 3, 128, 128)


# ---------------------------------------------------------------- GPTAQ drift correction
def _drift_problem(seed, T=60, n=10, m=3, drift=0.1):
    """Tiny layer with a drifted full-precision input: X, X~, and the damped H as the
    Gram matrix of X with sqrt(delta) I appended (X~ gets the same rows, so they carry no
    drift): H = X_aug^T X_aug = X^T X + delta I."""
    rng = _rng(seed)
    sc = np.exp(rng.standard_normal(n))
    X = rng.standard_normal((T, n)) * sc
    Xt = X + drift * rng.standard_normal((T, n)) * sc
    delta = 0.01 * np.mean(np.diag(X.T @ X))
    X_aug = np.vstack([X, np.sqrt(delta) * np.eye(n)])
    dX_aug = np.vstack([Xt - X, np.zeros((n, n))])
    H = ref.damp(X.T @ X, 0.01)
    W = rng.standard_normal((m, n)) * 0.05
    return X, Xt, X_aug, dX_aug, H, W


def test_drift_factor_brute_force_integers():
    """Delta X X^T of Algorithm 1 with tokens as rows: D[a, b] = sum_t (x~_t[a] - x_t[a]) x_t[b],
    by Python integer loops (D is not symmetric)."""
    rng = _rng(31)
    T, d = 23, 5
    X = rng.integers(-9, 10, size=(T, d))
    Xt = X + rng.integers(-3, 4, size=(T, d))
    D = ref.drift_factor(Xt.astype(np.float64), X.astype(np.float64))
    brute = [[sum(int(Xt[t, a] - X[t, a]) * int(X[t, b]) for t in range(T)) for b in range(d)]
             for a in range(d)]
    assert np.array_equal(D, np.array(brute, dtype=np.float64))
    assert not np.array_equal(D, D.T)


def test_p_rows_are_least_squares_projection_of_drift():
    """GPTAQ's sequential residual reading of Prop. 1: row p of P (alpha = 1) holds the
    least-squares coefficients of column p's drift Delta x_p on the later columns x_{p+1:},
    i.e. P[p, p+1:] = D[p, p+1:] H[p+1:, p+1:]^-1; P is strictly upper triangular and
    linear in alpha."""
    X, Xt, X_aug, dX_aug, H, _ = _drift_problem(41, n=12)
    n = H.shape[0]
    L = ref.lower_factor(H)
    P = ref.gptaq_p(ref.drift_factor(Xt, X), L, 1.0)
    assert np.all(np.tril(P) == 0)
    for p in range(n - 1):
        c, *_ = np.linalg.lstsq(X_aug[:, p + 1:], dX_aug[:, p], rcond=None)
        assert np.allclose(P[p, p + 1:], c, rtol=1e-9, atol=1e-12)
    P4 = ref.gptaq_p(ref.drift_factor(Xt, X), L, 0.25)
    assert np.allclose(P4, 0.25 * P, rtol=1e-12, atol=0)


@pytest.mark.parametrize("block", [3, 4, 16])
def test_sweep_with_p_is_sequential_residual_compensation(block):
    """Algorithm 2 with P (alpha = 1, per-row grid), blocked with a lazy trailing update,
    equals the column-by-column compensation of Prop. 1 restated as least squares: after
    quantizing column p, the later columns absorb the residual x_p (w_p - w^_p) + Delta x_p w_p
    (w_p the column's value just before quantization) by a least-squares fit on x_{p+1:}."""
    X, Xt, X_aug, dX_aug, H, W = _drift_problem(43, n=10)
    n = H.shape[0]
    R = ref.inverse_cholesky_upper(H)
    P = ref.gptaq_p(ref.drift_factor(Xt, X), R.T, 1.0)
    bits = 3
    sw = ref.obs_sweep(W, R, bits, 0, block, P)
    for r in range(W.shape[0]):
        s, z = ref.quant_params(W[r:r + 1], bits)
        v = W[r].copy()
        for p in range(n):
            assert np.isclose(sw["pre_q"][r, p], v[p], rtol=1e-9, atol=1e-12)
            q = ref.quantize(v[p], s[0], z[0], bits)
            assert sw["codes"][r, p] == q
            what = s[0] * (q - z[0])
            if p + 1 < n:
                resid = X_aug[:, p] * (v[p] - what) + dX_aug[:, p] * v[p]
                c, *_ = np.linalg.lstsq(X_aug[:, p + 1:], resid, rcond=None)
                v[p + 1:] += c


def test_zero_drift_gives_gptq_sweep():
    """X~ = X: D = 0, P = 0 and the sweep is the GPTQ-mode sweep, code for code."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=32, d_out=28, T=300)
    L = kqsynth.layer(cfg)
    a = ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], 3, 16, 16)
    b = ref.pipeline(L["X"], L["G"], L["W"], L["sign_u"], L["sign_v"], 3, 16, 16, Xt=L["X"])
    assert np.all(b["D"] == 0) and np.all(b["P"] == 0)
    assert np.array_equal(a["codes"], b["codes"])


def test_theorem1_invariance_with_drift_term():
    """Theorem 1 (both terms, appendix proof): the full objective of Eq. (kronq_full) is the
    same in the original space and after BiIP, with D carried as V S_X^-1 D S_X^-1 V^T."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=32, d_out=28, T=300)
    L = kqsynth.layer(cfg)
    Xt = kqsynth.fp_activations(cfg, L["X"])
    HX, HG = ref.accum_factor(L["X"]), ref.accum_factor(L["G"])
    D = ref.drift_factor(Xt, L["X"])
    W = L["W"].astype(np.float64)
    What = W + _rng(3).standard_normal(W.shape) * 0.01
    b = ref.biip(W, HX, HG, L["sign_u"], L["sign_v"], D)
    Whatp = b["U"] @ (b["s_g"][:, None] * What * b["s_x"][None, :]) @ b["V"].T
    j0 = ref.objective(W, What, HX, HG, D)
    j1 = ref.objective(b["W"], Whatp, b["HX"], b["HG"], b["D"])
    assert np.isclose(j0, j1, rtol=1e-9)
    # the drift term is really present: dropping it changes the value
    assert not np.isclose(j0, ref.objective(W, What, HX, HG), rtol=1e-6)
    # and the plain expansion of Eq. (gptaq_obj) with H_G = I: ||W X~^T - W^ X^T||^2 minus the
    # constant ||W (X~ - X)^T||^2
    Xd, Xtd = L["X"].astype(np.float64), Xt.astype(np.float64)
    full = np.sum((W @ Xtd.T - What @ Xd.T) ** 2) - np.sum((W @ (Xtd - Xd).T) ** 2)
    assert np.isclose(ref.objective(W, What, HX, np.eye(W.shape[0]), D), full, rtol=1e-9)


@pytest.mark.parametrize("group", [0, 32])
def test_fp32_sweep_with_p_matches_fp64_off_ties(group):
    """The fp32-ordered sweep with P agrees with the fp64 sweep wherever the decision is
    not within fp32 noise of a rounding tie."""
    X, Xt, _, _, H, _ = _drift_problem(47, T=400, n=64)
    R = ref.inverse_cholesky_upper(H)
    P = ref.gptaq_p(ref.drift_factor(Xt, X), R.T, 0.25)
    R32, P32 = R.astype(np.float32), P.astype(np.float32)
    W32 = (_rng(8).standard_normal((40, 64)) * 0.02).astype(np.float32)
    s64 = ref.obs_sweep(W32.astype(np.float64), R32.astype(np.float64), 4, group, 32,
                        P32.astype(np.float64))
    s32 = obs_sweep_fp32(W32, R32.T, 4, group, 32, Pt=P32.T)
    diff = s64["codes"] != s32["codes"]
    for r in np.nonzero(diff.any(1))[0]:
        j = np.argmax(diff[r])
        g = 0 if group == 0 else j // group
        t = s64["pre_q"][r, j] / s64["scale"][r, g]
        assert abs(abs(t - np.floor(t)) - 0.5) < 1e-3
    assert diff.mean() < 0.02
    # P really changes the result
    s0 = obs_sweep_fp32(W32, R32.T, 4, group, 32)
    assert not np.array_equal(s0["codes"], s32["codes"])


# ------------------------------------------------------- mixed-precision allocation
def test_allocation_worked_examples_golden():
    """Hand-worked W2 -> W3 allocations (tests/golden/mp_allocation_worked.json)."""
    g = json.load(open(os.path.join(GOLDEN, "mp_allocation_worked.json")))
    for c in g["cases"]:
        assert ref.allocate_bits(c["scores"], c["params"], g["low"], g["high"], c["budget"]) == c["bits"], c["work"]


def test_allocation_limits_and_monotone_budget():
    rng = _rng(12)
    names = [f"s{i}" for i in range(7)]
    scores = dict(zip(names, rng.random(7)))
    params = dict(zip(names, rng.integers(1, 20, 7).tolist()))
    assert set(ref.allocate_bits(scores, params, 2, 3, 2.0).values()) == {2}
    assert set(ref.allocate_bits(scores, params, 2, 3, 3.0).values()) == {3}
    prev = set()
    for budget in np.linspace(2.0, 3.0, 41):
        b = ref.allocate_bits(scores, params, 2, 3, budget)
        up = {n for n in names if b[n] == 3}
        assert prev <= up                           # a larger budget never downgrades
        mean = sum(b[n] * params[n] for n in names) / sum(params.values())
        assert mean <= budget + 1e-12
        # the upgraded set is a prefix of the descending-score order
        order = sorted(names, key=lambda n: -scores[n])
        assert up == set(order[:len(up)])
        prev = up


def test_block_scores_shared_input_degeneracy():
    """Sec. 3.3: q, k, v read the same input, so every activation-only score (raw tr(H_X))
    is identical for them; the joint score differs through tr(H_G)."""
    cfg = kqsynth.BLOCKS["tiny_block"].replace(T=256)
    b = kqsynth.block_inputs(cfg)
    sc = ref.block_scores(b["X"], b["G"], b["W"], kqsynth.block_spec(cfg))
    assert sc["q"]["trHX"] == sc["k"]["trHX"] == sc["v"]["trHX"]
    assert sc["gate"]["trHX"] == sc["up"]["trHX"]
    assert len({sc[n]["trHG"] for n in ("q", "k", "v")}) == 3
    for n, v in sc.items():
        assert np.isclose(v["s"], v["trHX"] * v["trHG"], rtol=1e-12)
        # post-BiIP traces follow the rescale identity sum_j h_j / s_j^2 (checked against
        # the dense rotated factor of that sublayer)
    name, grp, _, _ = kqsynth.block_spec(cfg)[1]
    su, sv = b["sign_u"][name], b["sign_v"][name]
    r = ref.biip(b["W"][name], ref.accum_factor(b["X"][grp]), ref.accum_factor(b["G"][name]), su, sv)
    assert np.isclose(np.trace(r["HX"]), sc[name]["trHX_post"], rtol=1e-10)
    assert np.isclose(np.trace(r["HG"]), sc[name]["trHG_post"], rtol=1e-10)


# ------------------------------------------------------------------------ inference
def test_infer_reproduces_the_layer_within_the_grid_bound():
    """8-bit per-row codes of W' = U S_G W S_X V^T reverted and applied to tokens give W x
    up to the rounding of the grid: |W^ - W| is the reverted error of |Q' - W'| <= scale / 2
    (rotations are orthogonal, so ||(W^ - W) x|| <= ||S_G^-1|| ||Q' - W'||_2 ||S_X^-1 x||)."""
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_out=64, d_in=128, T=512)
    L = kqsynth.layer(cfg)
    HX, HG = ref.accum_factor(L["X"]), ref.accum_factor(L["G"])
    b = ref.biip(L["W"], HX, HG, L["sign_u"], L["sign_v"])
    s, z = ref.quant_params(b["W"], 8)
    codes = ref.quantize(b["W"], s[:, None], z[:, None], 8).astype(np.uint8)
    x = _rng(4).standard_normal((3, 128))
    y = ref.infer(codes, s[:, None], z[:, None], 0, b["s_x"], b["s_g"], L["sign_u"], L["sign_v"], x)
    W = L["W"].astype(np.float64)
    dWp = ref.dequant(codes, s[:, None], z[:, None], 0) - b["W"]
    assert np.max(np.abs(dWp) / s[:, None]) <= 0.5 + 1e-9
    bound = np.linalg.norm(dWp, 2) / np.min(b["s_g"]) * np.linalg.norm(x / b["s_x"][None, :], axis=1)
    err = np.linalg.norm(y - x @ W.T, axis=1)
    assert np.all(err <= bound * (1 + 1e-9))
    assert np.all(err > 0)


# --------------------------------------------------------------- BiIP statistics (Prop. 2)
def test_norm_cv_closed_forms():
    """Columns with norms 1, 2, 3, 4 (and rows all equal): CV_in = std/mean of (1, 2, 3, 4)
    = sqrt(1.25) / 2.5; CV_out = 0."""
    W = np.zeros((4, 4))
    for j, nrm in enumerate([1.0, 2.0, 3.0, 4.0]):
        W[:, j] = nrm / 2.0             # each column: four entries of nrm / 2 -> norm nrm
    W = W[:, [0, 1, 2, 3]]
    cv_in, cv_out = ref.norm_cv(W)
    assert np.isclose(cv_in, np.sqrt(1.25) / 2.5, rtol=1e-12)
    assert np.isclose(cv_out, 0.0, atol=1e-15)
    # orthogonal rotations on the column side keep every row norm (CV_out unchanged)
    Wr = np.random.default_rng(0).standard_normal((16, 32)) * np.exp(np.linspace(0, 3, 32))
    V = ref.rht_matrix(32, np.ones(32))
    assert np.isclose(ref.norm_cv(Wr @ V.T)[1], ref.norm_cv(Wr)[1], rtol=1e-12)


def test_rho_bounds_and_equality():
    """rho <= 1 (Cauchy-Schwarz), = 1 iff h is proportional to a, ~k/d when the curvature sits
    on k channels of equal row energy (the appendix's concentration remark)."""
    rng = _rng(14)
    h, a = rng.random(50) + 0.01, rng.random(50) + 0.01
    assert ref.rho(h, a) < 1.0
    assert np.isclose(ref.rho(3.0 * a, a), 1.0, rtol=1e-14)
    d, k = 1000, 10
    hk = np.zeros(d)
    hk[:k] = 1.0
    assert np.isclose(ref.rho(hk, np.ones(d)), k / d, rtol=1e-12)


def test_prop2_bound_minimized_at_quarter_exponent():
    """Prop. 2: over s = (h/a)^alpha the factor (sum h/s^2)(sum s^2 a) is smallest at
    alpha = 1/4, where it equals (sum sqrt(h a))^2; a fine sweep finds the minimum there."""
    rng = _rng(15)
    h = np.exp(rng.standard_normal(200) * 1.5)
    a = np.exp(rng.standard_normal(200) * 0.7)
    alphas = np.linspace(0.0, 0.5, 201)
    vals = [ref.prop2_bound(h, a, (h / a) ** al) for al in alphas]
    assert np.isclose(alphas[int(np.argmin(vals))], 0.25, atol=1e-9)
    assert np.isclose(min(vals), np.sum(np.sqrt(h * a)) ** 2, rtol=1e-12)
    assert np.isclose(vals[0] , np.sum(h) * np.sum(a), rtol=1e-12)          # alpha = 0: s = 1
    assert np.isclose(min(vals) / vals[0], ref.rho(h, a), rtol=1e-12)


def test_scales_exponent_quarter_is_the_paper_rescale():
    cfg = kqsynth.CONFIGS["tiny256"].replace(d_in=64, d_out=32, T=200)
    L = kqsynth.layer(cfg)
    HX, HG = ref.accum_factor(L["X"]), ref.accum_factor(L["G"])
    sx, sg = ref.biip_scales(L["W"], HX, HG)
    sx2, sg2 = ref.biip_scales_exp(L["W"], np.diag(HX), np.diag(HG), 0.25, 0.25)
    assert np.allclose(sx, sx2, rtol=1e-14) and np.allclose(sg, sg2, rtol=1e-14)
    sx0, sg0 = ref.biip_scales_exp(L["W"], np.diag(HX), np.diag(HG), 0.0, 0.0)
    assert np.all(sx0 == 1.0) and np.all(sg0 == 1.0)
