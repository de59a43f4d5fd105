"""Plain float64 CPU oracle of the KronQ per-layer quantization path.

TEST INFRASTRUCTURE ONLY. This module exists to check the CUDA library; only the tests,
the smoke check and the benchmark's CPU-baseline leg may import it. The product path
never calls it, and it shares no code with the CUDA kernels.

It follows "KronQ: LLM Quantization via Kronecker-Factored Hessian":
  * Kronecker factors          Sec. 2.1 Eq. (ptq_obj), Sec. 3.1 Eq. (kfac), Algorithm 1
  * bidirectional rescaling    Sec. 3.2 Eq. (rescale), Algorithm 1
  * randomized Hadamard (BiIP) Sec. 3.2 Eq. (biip), Algorithm 1
  * damping, inverse Cholesky  Algorithm 2, Proposition 1
  * column-wise OBS sweep      Sec. 2.1 Eq. (obs_update), Algorithm 2 (GPTQ mode, P = 0)
  * GPTAQ drift correction     Sec. 2.1 Eq. (gptaq_obj), Sec. 3.1 Eq. (kronq_full),
                               Proposition 1 (P), Algorithms 1 and 2 (Delta X X^T, P)
  * revert and proxy loss      Algorithm 2, Sec. 3.1 Eq. (kron_obj), Theorem 1
  * sensitivity traces         Sec. 3.3 Eq. (sensitivity)
  * mixed-precision allocation Sec. 3.3, Sec. 5 "Results on Mixed-precision" (W2 -> W3)
  * inference y = W^ x         Algorithm 2's revert applied to tokens (Sec. 3.2)
  * BiIP statistics            Prop. 2 (rho, the exponent of the rescale), Sec. 3.2 and
                               the appendix on weight distributions (CV_in, CV_out)
Tokens are stored as rows here (X is T x d_in), so the paper's X X^T is X^T X.

Readings of points the paper leaves open (all listed in the design notes):
  * factors are raw sums over tokens (no 1/T);
  * the rotations are V = H_n diag(sigma_V) / sqrt(n) with H_n Sylvester for n = 2^k and
    H_28 (Paley construction II, q = 13) Kronecker H_{2^k} for n = 28 * 2^k;
  * damping adds damp * mean(diag) to the rescaled, rotated H_X;
  * the update row of Algorithm 2 is row j of R = L^T, H^-1 = R^T R (R upper);
  * the quantizer is the asymmetric min-max grid of GPTQ/GPTAQ with round-half-even;
  * per-row grids come from the whole rotated row before the sweep; group grids
    (group == block) from the current, compensated block at block start;
  * the per-column loss is sum over rows of E_j^2 (no 1/2);
  * the drift statistic is D = (X~ - X)^T X (tokens as rows), transformed like H_X;
  * W_{:,j} in the P terms of Proposition 1 and Algorithm 2 is column j's value just
    before it is quantized, in the column update and in the lazy trailing update alike;
  * the W2 -> W3 allocation upgrades sublayers in descending post-BiIP score while the
    parameter-weighted mean bit width stays within the budget, stopping at the first
    upgrade that would exceed it (ties keep the listed order).
"""
from __future__ import annotations

import numpy as np

__all__ = [
    "accum_factor", "biip_scales_from_diag", "sylvester", "paley28", "hadamard_matrix", "rht_matrix",
    "biip_scales", "biip", "damp", "inverse_cholesky_upper", "lower_factor", "lower_factor_reversed",
    "quant_params", "quantize", "quantize_f32", "teacher_forced", "obs_sweep", "dequant", "revert", "proxy_loss",
    "traces", "pipeline", "drift_factor", "gptaq_p", "objective", "allocate_bits", "block_scores",
    "block_pipeline", "infer", "biip_scales_exp", "norm_cv", "rho", "prop2_bound",
]


# ----------------------------------------------------------------------------------
# Stage 1: Kronecker factors (Eq. ptq_obj: H_X = X X^T; Eq. kfac: H_G = E[g g^T];
# Algorithm 1, "online statistics").
# ----------------------------------------------------------------------------------
def accum_factor(A: np.ndarray) -> np.ndarray:
    """H = A^T A for A [T, d] with tokens as rows, in float64 (a library matmul)."""
    A = np.asarray(A, dtype=np.float64)
    return A.T @ A


def drift_factor(Xt, X) -> np.ndarray:
    """Algorithm 1's drift statistic Delta X X^T = (X~ - X) X^T, with tokens as rows here:
    D = (X~ - X)^T X, D[a, b] = sum_t (x~_t[a] - x_t[a]) x_t[b] (not symmetric). X~ is the
    full-precision model's input to the layer, X the running quantized model's (Sec. 2.1,
    Eq. gptaq_obj)."""
    Xt = np.asarray(Xt, dtype=np.float64)
    X = np.asarray(X, dtype=np.float64)
    return (Xt - X).T @ X


# ----------------------------------------------------------------------------------
# Randomized Hadamard transforms (Eq. biip; Algorithm 1 "sample random Hadamard").
# ----------------------------------------------------------------------------------
def sylvester(n: int) -> np.ndarray:
    """Sylvester Hadamard matrix of order n = 2^k (H_2 = [[1, 1], [1, -1]], H_2n = H_2 (x) H_n)."""
    if n < 1 or n & (n - 1):
        raise ValueError(f"{n} is not a power of two")
    h = np.ones((1, 1), dtype=np.int64)
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


def paley28() -> np.ndarray:
    """Hadamard matrix of order 28 by Paley's second construction with q = 13.

    chi is the quadratic character of GF(13); the Jacobsthal matrix Q[i, j] = chi(j - i)
    is symmetric because 13 = 1 (mod 4). The conference matrix C = [[0, 1^T], [1, Q]] of
    order 14 is expanded entry by entry: 0 -> [[1, -1], [-1, -1]], +-1 -> +-[[1, 1], [1, -1]].
    """
    q = 13
    squares = {(x * x) % q for x in range(1, q)}

    def chi(a: int) -> int:
        a %= q
        return 0 if a == 0 else (1 if a in squares else -1)

    C = np.zeros((q + 1, q + 1), dtype=np.int64)
    C[0, 1:] = 1
    C[1:, 0] = 1
    for i in range(q):
        for j in range(q):
            C[1 + i, 1 + j] = chi(j - i)
    zero_blk = np.array([[1, -1], [-1, -1]], dtype=np.int64)
    one_blk = np.array([[1, 1], [1, -1]], dtype=np.int64)
    H = np.zeros((2 * (q + 1), 2 * (q + 1)), dtype=np.int64)
    for i in range(q + 1):
        for j in range(q + 1):
            H[2 * i:2 * i + 2, 2 * j:2 * j + 2] = zero_blk if C[i, j] == 0 else C[i, j] * one_blk
    return H


def hadamard_matrix(n: int) -> np.ndarray:
    """H_n for n = 2^k (Sylvester) or n = 28 * 2^k (H_28 (x) H_{2^k}, index a * 2^k + b)."""
    if n >= 1 and n & (n - 1) == 0:
        return sylvester(n)
    if n % 28 == 0 and (n // 28) & (n // 28 - 1) == 0:
        return np.kron(paley28(), sylvester(n // 28))
    raise ValueError(f"no Hadamard construction for n = {n}")


def rht_matrix(n: int, sign: np.ndarray) -> np.ndarray:
    """Randomized Hadamard transform V = H_n diag(sigma) / sqrt(n) (orthogonal)."""
    sign = np.asarray(sign, dtype=np.float64).reshape(-1)
    assert sign.shape == (n,)
    return hadamard_matrix(n).astype(np.float64) * sign[None, :] / np.sqrt(n)


def rht_rows(n: int, sign: np.ndarray, rows) -> np.ndarray:
    """Selected rows of V = H_n diag(sigma) / sqrt(n) without forming H_n (for sizes where the
    dense n x n matrix is too large): Sylvester entries are (-1)^popcount(i & j); for
    n = 28 * 2^k, H_n[i, j] = H_28[i // 2^k, j // 2^k] * H_{2^k}[i % 2^k, j % 2^k]."""
    sign = np.asarray(sign, dtype=np.float64).reshape(-1)
    assert sign.shape == (n,)
    rows = np.asarray(rows, dtype=np.int64).reshape(-1)
    if n >= 1 and n & (n - 1) == 0:
        P, h28 = n, None
    elif n % 28 == 0 and (n // 28) & (n // 28 - 1) == 0:
        P, h28 = n // 28, paley28()
    else:
        raise ValueError(f"no Hadamard construction for n = {n}")
    j = np.arange(n, dtype=np.int64)
    out = np.empty((len(rows), n), dtype=np.float64)
    for t, i in enumerate(rows):
        both = (i % P) & (j % P)
        parity = np.zeros(n, dtype=np.int64)
        while np.any(both):
            parity ^= both & 1
            both >>= 1
        v = 1.0 - 2.0 * parity
        if h28 is not None:
            v = v * h28[i // P, j // P]
        out[t] = v * sign / np.sqrt(n)
    return out


# ----------------------------------------------------------------------------------
# Stage 2: bidirectional incoherence processing (Eq. rescale, Eq. biip, Algorithm 1).
# ----------------------------------------------------------------------------------
def biip_scales(W: np.ndarray, HX: np.ndarray, HG: np.ndarray):
    """S_X = (diag(H_X) / diag(W^T W))^(1/4), S_G = (diag(H_G) / diag(W W^T))^(1/4).

    A channel whose Hessian diagonal or weight norm is zero gets scale 1 (reading of a
    case the paper does not discuss).
    """
    W = np.asarray(W, dtype=np.float64)
    a = np.sum(W * W, axis=0)          # ||W_{:,j}||^2, j over d_in
    r = np.sum(W * W, axis=1)          # ||W_{i,:}||^2, i over d_out
    hx = np.diag(HX).astype(np.float64)
    hg = np.diag(HG).astype(np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        sx = np.where((hx > 0) & (a > 0), (hx / a) ** 0.25, 1.0)
        sg = np.where((hg > 0) & (r > 0), (hg / r) ** 0.25, 1.0)
    return sx, sg


def biip_scales_from_diag(W: np.ndarray, hx: np.ndarray, hg: np.ndarray):
    """Eq. (rescale) from the factors' diagonals alone (all that the scales read)."""
    return biip_scales(W, np.diag(np.asarray(hx, np.float64)), np.diag(np.asarray(hg, np.float64)))


def biip(W, HX, HG, sign_u, sign_v, D=None, ex: float = 0.25, eg: float = 0.25):
    """Algorithm 1: W <- S_G W S_X; H_X <- S_X^-1 H_X S_X^-1; H_G <- S_G^-1 H_G S_G^-1;
    W <- U W V^T; H_X <- V H_X V^T; H_G <- U H_G U^T (dense products). With the drift
    statistic D (Delta X X^T), also D <- V S_X^-1 D S_X^-1 V^T. ex, eg: the rescale's
    exponents (1/4 in Eq. rescale; Prop. 2's sweep varies them)."""
    W = np.asarray(W, dtype=np.float64)
    HX = np.asarray(HX, dtype=np.float64)
    HG = np.asarray(HG, dtype=np.float64)
    d_out, d_in = W.shape
    if ex == 0.25 and eg == 0.25:
        sx, sg = biip_scales(W, HX, HG)
    else:
        sx, sg = biip_scales_exp(W, np.diag(HX), np.diag(HG), ex, eg)
    Ws = sg[:, None] * W * sx[None, :]
    HXs = HX / sx[:, None] / sx[None, :]
    HGs = HG / sg[:, None] / sg[None, :]
    U = rht_matrix(d_out, sign_u)
    V = rht_matrix(d_in, sign_v)
    out = {"W": U @ Ws @ V.T, "HX": V @ HXs @ V.T, "HG": U @ HGs @ U.T,
           "s_x": sx, "s_g": sg, "U": U, "V": V}
    if D is not None:
        Ds = np.asarray(D, dtype=np.float64) / sx[:, None] / sx[None, :]
        out["D"] = V @ Ds @ V.T
    return out


# ----------------------------------------------------------------------------------
# Stage 3: damping and inverse Cholesky (Algorithm 2; Proposition 1 names L with
# H_X^-1 = L L^T).
# ----------------------------------------------------------------------------------
def damp(H: np.ndarray, lam: float) -> np.ndarray:
    """H + lam * mean(diag(H)) * I."""
    H = np.asarray(H, dtype=np.float64)
    return H + lam * np.mean(np.diag(H)) * np.eye(H.shape[0])


def inverse_cholesky_upper(Hd: np.ndarray) -> np.ndarray:
    """R upper triangular with positive diagonal and Hd^-1 = R^T R, by the textbook
    route: a library inverse followed by a library Cholesky."""
    Hinv = np.linalg.inv(np.asarray(Hd, dtype=np.float64))
    Hinv = 0.5 * (Hinv + Hinv.T)
    return np.linalg.cholesky(Hinv).T


def lower_factor(Hd: np.ndarray) -> np.ndarray:
    """The paper's L = R^T (lower), H^-1 = L L^T; this is what kq_chol_inv returns."""
    return inverse_cholesky_upper(Hd).T


def lower_factor_reversed(Hd: np.ndarray, panel: int = 2048) -> np.ndarray:
    """The same L (H^-1 = L L^T, L lower with a positive diagonal, which is unique) by the
    cheaper route for large n: the Cholesky factor C of the reversed matrix J H J (J the
    exchange matrix) gives H = (J C J)(J C J)^T with J C J upper, so H^-1 = R^T R for
    R = (J C J)^-1, and L = R^T = J C^-T J. Library Cholesky (LAPACK dpotrf), then C^-1 one
    panel of columns at a time by triangular solves (BLAS dtrsm) on the rows at and below
    the panel (C^-1 is lower triangular): about 2 n^3 / 3 flops instead of the textbook
    route's ~3 n^3."""
    from scipy.linalg import blas, lapack
    n = np.asarray(Hd).shape[0]
    A = np.asfortranarray(np.asarray(Hd, dtype=np.float64)[::-1, ::-1])
    C, info = lapack.dpotrf(A, lower=1, clean=1, overwrite_a=1)
    if info != 0:
        raise np.linalg.LinAlgError(f"dpotrf failed ({info})")
    Ci = np.zeros((n, n), order="F")
    for j0 in range(0, n, panel):
        j1 = min(n, j0 + panel)
        rhs = np.zeros((n - j0, j1 - j0), order="F")
        rhs[np.arange(j1 - j0), np.arange(j1 - j0)] = 1.0
        Ci[j0:, j0:j1] = blas.dtrsm(1.0, np.asfortranarray(C[j0:, j0:]), rhs, lower=1, overwrite_b=1)
    return np.ascontiguousarray(Ci.T[::-1, ::-1])


def gptaq_p(Dp: np.ndarray, L: np.ndarray, alpha: float) -> np.ndarray:
    """The GPTAQ correction of Proposition 1 and Algorithm 2:
    P = alpha ((D' L) o M_U) L^T, with D' the rescaled, rotated drift statistic, L the
    lower factor of the damped H^-1 = L L^T and M_U the strictly upper-triangular mask.
    P is strictly upper triangular."""
    Dp = np.asarray(Dp, dtype=np.float64)
    L = np.asarray(L, dtype=np.float64)
    n = L.shape[0]
    M_U = np.triu(np.ones((n, n)), 1)
    return alpha * ((Dp @ L) * M_U) @ L.T


# ----------------------------------------------------------------------------------
# Stage 4: quantizer and the blocked OBS sweep (Eq. obs_update, Algorithm 2 with P = 0).
# ----------------------------------------------------------------------------------
def quant_params(x: np.ndarray, bits: int):
    """Asymmetric min-max grid per row of x: xmin = min(0, min x), xmax = max(0, max x),
    (-1, 1) when both are 0; scale = (xmax - xmin) / (2^b - 1); zero = rint(-xmin/scale)."""
    x = np.asarray(x, dtype=np.float64)
    xmin = np.minimum(x.min(axis=-1), 0.0)
    xmax = np.maximum(x.max(axis=-1), 0.0)
    both = (xmin == 0) & (xmax == 0)
    xmin = np.where(both, -1.0, xmin)
    xmax = np.where(both, 1.0, xmax)
    scale = (xmax - xmin) / (2 ** bits - 1)
    zero = np.rint(-xmin / scale)
    return scale, zero


def quantize(w, scale, zero, bits):
    """q = clamp(rint(w / scale) + zero, 0, 2^b - 1) (round half to even)."""
    return np.clip(np.rint(np.asarray(w, np.float64) / scale) + zero, 0, 2 ** bits - 1)


def obs_sweep(Wp: np.ndarray, R: np.ndarray, bits: int, group: int, block: int, P=None):
    """Column-wise OBS sweep of Algorithm 2; GPTQ mode when P is None.

    For each block [i, e): for j in the block, quantize column j, E_j = (w_j - w^_j)/R_jj,
    update the rest of the block by -E_j R[j, j+1:e] + w_j P[j, j+1:e]; then the lazy
    trailing update W[:, e:] -= E_blk R[i:e, e:] - Wpre_blk P[i:e, e:], where w_j and Wpre
    are the columns' values just before they were quantized (Proposition 1's W_{:,p}).
    Returns codes, scale, zero (per row or per group) and E for every column (the
    per-column loss is sum over rows of E^2), and pre_q, the value of each column just
    before it is quantized.
    """
    W = np.array(Wp, dtype=np.float64, copy=True)
    R = np.asarray(R, dtype=np.float64)
    if P is not None:
        P = np.asarray(P, dtype=np.float64)
    m, n = W.shape
    if group not in (0, block):
        raise ValueError("group must be 0 (per row) or equal to the block size")
    ngroups = 1 if group == 0 else (n + group - 1) // group
    codes = np.zeros((m, n), dtype=np.uint8)
    scale = np.zeros((m, ngroups))
    zero = np.zeros((m, ngroups))
    E = np.zeros((m, n))
    pre_q = np.zeros((m, n))
    if group == 0:
        s, z = quant_params(W, bits)
        scale[:, 0], zero[:, 0] = s, z
    for i in range(0, n, block):
        e = min(i + block, n)
        if group:
            s, z = quant_params(W[:, i:e], bits)
            scale[:, i // group], zero[:, i // group] = s, z
        gidx = 0 if group == 0 else i // group
        for j in range(i, e):
            w = W[:, j]
            pre_q[:, j] = w
            q = quantize(w, scale[:, gidx], zero[:, gidx], bits)
            codes[:, j] = q.astype(np.uint8)
            what = scale[:, gidx] * (q - zero[:, gidx])
            E[:, j] = (w - what) / R[j, j]
            W[:, j + 1:e] -= np.outer(E[:, j], R[j, j + 1:e])
            if P is not None:
                W[:, j + 1:e] += np.outer(pre_q[:, j], P[j, j + 1:e])
        if e < n:
            W[:, e:] -= E[:, i:e] @ R[i:e, e:]
            if P is not None:
                W[:, e:] += pre_q[:, i:e] @ P[i:e, e:]
    return {"codes": codes, "scale": scale, "zero": zero, "E": E, "pre_q": pre_q}


def quantize_f32(w, scale, zero, bits):
    """The column step's rounding in float32, as Algorithm 2 runs in a float32 sweep:
    q = clamp(rint(w / scale) + zero, 0, 2^b - 1) with w / scale one correctly rounded
    float32 division and rint half to even (not rint(w / scale + zero): the two differ at
    ties when zero is odd)."""
    w = np.asarray(w, np.float32)
    scale = np.asarray(scale, np.float32)
    zero = np.asarray(zero, np.float32)
    q = np.rint(w / scale) + zero
    return np.clip(q, np.float32(0), np.float32(2 ** bits - 1)).astype(np.uint8)


def _strict_lower64(M) -> np.ndarray:
    """float64 copy of M with the diagonal and everything above it zeroed (row slabs, so
    that a large M needs no index arrays)."""
    out = np.array(M, dtype=np.float64)
    for i0 in range(0, out.shape[0], 1024):
        out[i0:i0 + 1024] = np.tril(out[i0:i0 + 1024], i0 - 1)
    return out


def teacher_forced(Wp, Lt, pre_q, codes, scale, zero, bits: int, group: int, block: int = 128, Pt=None) -> dict:
    """Algorithm 2 replayed on another sweep's own decisions (teacher forcing), for rows of
    a layer given that sweep's outputs: its pre-quantization values pre_q, codes and grids
    (float32), the rotated weights W' it started from and Lt = R^T (and Pt = P^T with the
    GPTAQ correction).

    Each column step fixes the error from the column's own value and code,
        E_j = (w_j - scale (q_j - zero)) / R_jj           (float32, as the sweep computes it),
    and every later column then sees the same compensation Algorithm 2 applies (Eq.
    obs_update, with the lazy block updates summed out):
        w_j = W'_j - sum_{k < j} E_k R_kj (+ sum_{k < j} w_k P_kj),
    evaluated here in float64 from those errors. A sweep that computes what Algorithm 2
    states quantizes, at column j, a value within its float32 rounding of w_j, and its code
    is exactly the float32 quantization of its own value. Returned:
      E         the errors (float32),
      pre_q     w_j in float64,
      codes     quantize_f32 of the given pre_q on the given grid (what the codes must be),
      absum     |W'_j| + sum_{k < j} |E_k R_kj| (+ |w_k P_kj|): the scale of w_j's rounding,
      block_start (group = block) the columns' float64 values at their block's start,
                W'_c - sum_{k < block start} E_k R_kc (+ P terms), from which the group grid
                is drawn (Sec. 5.1 grids, group statistics at the block start).
    Rows are independent given R, so any subset of rows can be passed."""
    Wp = np.asarray(Wp, np.float64)
    m, n = Wp.shape
    pq32 = np.asarray(pre_q, np.float32)
    sc = np.asarray(scale, np.float32)
    zr = np.asarray(zero, np.float32)
    ng = sc.shape[1]
    gidx = np.zeros(n, np.int64) if group == 0 else np.arange(n) // group
    s_col = sc[:, gidx] if ng > 1 else np.repeat(sc, n, axis=1)
    z_col = zr[:, gidx] if ng > 1 else np.repeat(zr, n, axis=1)
    q = np.asarray(codes, np.float32)
    diag = np.ascontiguousarray(np.diagonal(np.asarray(Lt, np.float32)))
    what = s_col * (q - z_col)
    E = (pq32 - what) / diag[None, :]
    Ls = _strict_lower64(Lt)                                # R_kj (k < j) at Ls[j, k]
    E64 = E.astype(np.float64)
    comp = E64 @ Ls.T                                       # sum_{k < j} E_k R_kj
    absum = np.abs(Wp) + np.abs(E64) @ np.abs(Ls).T
    if Pt is not None:
        Ps = _strict_lower64(Pt)                            # P_kj (k < j) at Ps[j, k]
        comp -= pq32.astype(np.float64) @ Ps.T
        absum += np.abs(pq32.astype(np.float64)) @ np.abs(Ps).T
    out = {"E": E, "pre_q": Wp - comp, "codes": quantize_f32(pq32, s_col, z_col, bits), "absum": absum}
    if group:
        # add back the in-block part of the compensation: the values at the block's start
        bs = out["pre_q"].copy()
        for i in range(0, n, block):
            e = min(i + block, n)
            blk = Ls[i:e, i:e]
            bs[:, i:e] += E64[:, i:e] @ blk.T
            if Pt is not None:
                bs[:, i:e] -= pq32[:, i:e].astype(np.float64) @ Ps[i:e, i:e].T
        out["block_start"] = bs
    return out


def dequant(codes, scale, zero, group: int) -> np.ndarray:
    """Q' = scale * (q - zero) on the grid of each row or group."""
    codes = np.asarray(codes, dtype=np.float64)
    m, n = codes.shape
    if group == 0:
        return scale[:, :1] * (codes - zero[:, :1])
    gi = np.arange(n) // group
    return scale[:, gi] * (codes - zero[:, gi])


def revert(Qp, s_x, s_g, U, V) -> np.ndarray:
    """Algorithm 2's revert: Q <- U^T Q V, then Q <- S_G^-1 Q S_X^-1."""
    Q = U.T @ np.asarray(Qp, dtype=np.float64) @ V
    return Q / s_g[:, None] / s_x[None, :]


def proxy_loss(W, What, HX, HG) -> float:
    """tr(H_G dW H_X dW^T) with dW = W - W^ (Eq. kron_obj)."""
    dW = np.asarray(W, np.float64) - np.asarray(What, np.float64)
    return float(np.trace(np.asarray(HG, np.float64) @ dW @ np.asarray(HX, np.float64) @ dW.T))


def objective(W, What, HX, HG, D=None) -> float:
    """The full objective of Eq. (kronq_full): tr[H_G (dW H_X dW^T + 2 W D dW^T)], dW = W - W^,
    D = Delta X X^T (the second term is absent when D is None)."""
    W = np.asarray(W, np.float64)
    dW = W - np.asarray(What, np.float64)
    HG = np.asarray(HG, np.float64)
    val = np.trace(HG @ dW @ np.asarray(HX, np.float64) @ dW.T)
    if D is not None:
        val += 2.0 * np.trace(HG @ W @ np.asarray(D, np.float64) @ dW.T)
    return float(val)


def traces(HX, HG, HXp, HGp) -> dict:
    """Sensitivity s = tr(H_G) tr(H_X) (Eq. sensitivity), raw and after BiIP."""
    tx, tg = float(np.trace(HX)), float(np.trace(HG))
    txp, tgp = float(np.trace(HXp)), float(np.trace(HGp))
    return {"trHX": tx, "trHG": tg, "s": tx * tg, "trHX_post": txp, "trHG_post": tgp,
            "s_post": txp * tgp}


def pipeline(X, G, W, sign_u, sign_v, bits: int, group: int, block: int = 128,
             lam: float = 0.01, Xt=None, alpha: float = 0.25, ex: float = 0.25, eg: float = 0.25) -> dict:
    """Algorithms 1 and 2 end to end, all in float64: GPTQ mode when Xt (X~) is None,
    else with the GPTAQ drift correction P of scaling alpha; ex, eg the rescale exponents."""
    HX = accum_factor(X)
    HG = accum_factor(G)
    D = None if Xt is None else drift_factor(Xt, X)
    b = biip(W, HX, HG, sign_u, sign_v, D, ex, eg)
    Hd = damp(b["HX"], lam)
    R = inverse_cholesky_upper(Hd)
    P = None if D is None else gptaq_p(b["D"], R.T, alpha)
    sw = obs_sweep(b["W"], R, bits, group, block, P)
    Qp = dequant(sw["codes"], sw["scale"], sw["zero"], group)
    What = revert(Qp, b["s_x"], b["s_g"], b["U"], b["V"])
    out = {"HX": HX, "HG": HG, "Wp": b["W"], "HXp": b["HX"], "HGp": b["HG"],
           "s_x": b["s_x"], "s_g": b["s_g"], "Hd": Hd, "R": R, "L": R.T,
           "What": What, "loss": proxy_loss(W, What, HX, HG),
           "loss_rot": proxy_loss(b["W"], Qp, b["HX"], b["HG"]),
           "col_loss": np.sum(sw["E"] ** 2, axis=0)}
    if D is not None:
        out.update({"D": D, "Dp": b["D"], "P": P, "objective": objective(W, What, HX, HG, D)})
    out.update(sw)
    out.update(traces(HX, HG, b["HX"], b["HG"]))
    return out


# ----------------------------------------------------------------------------------
# Mixed-precision allocation across the sublayers of a block (Sec. 3.3 Eq. sensitivity;
# Sec. 5 "Results on Mixed-precision": the most sensitive sublayers go from W2 to W3).
# ----------------------------------------------------------------------------------
def allocate_bits(scores: dict, params: dict, low: int, high: int, budget: float) -> dict:
    """Upgrade sublayers from `low` to `high` bits in descending score, one at a time, while
    the parameter-weighted mean bit width sum(bits * params) / sum(params) stays within
    `budget`; the first upgrade that would exceed it ends the allocation. Equal scores keep
    the order of `scores`."""
    names = list(scores)
    order = sorted(range(len(names)), key=lambda i: -scores[names[i]])   # stable
    total = float(sum(params[n] for n in names))
    bits = {n: low for n in names}
    used = low * total
    for i in order:
        n = names[i]
        if (used + (high - low) * params[n]) / total > budget:
            break
        bits[n] = high
        used += (high - low) * params[n]
    return bits


def block_scores(X: dict, G: dict, W: dict, spec) -> dict:
    """Per sublayer: raw and post-BiIP traces and the sensitivity s = tr(H_G) tr(H_X)
    (Eq. sensitivity, computed post-BiIP). spec lists (name, input group, d_out, d_in);
    sublayers of one input group share H_X."""
    HX = {g: accum_factor(X[g]) for g in {grp for _, grp, _, _ in spec}}
    out = {}
    for name, grp, _, _ in spec:
        HG = accum_factor(G[name])
        sx, sg = biip_scales(W[name], HX[grp], HG)
        hx, hg = np.diag(HX[grp]), np.diag(HG)
        out[name] = {"trHX": float(np.sum(hx)), "trHG": float(np.sum(hg)),
                     "trHX_post": float(np.sum(hx / sx ** 2)), "trHG_post": float(np.sum(hg / sg ** 2))}
        out[name]["s"] = out[name]["trHX"] * out[name]["trHG"]
        out[name]["s_post"] = out[name]["trHX_post"] * out[name]["trHG_post"]
    return out


def block_pipeline(X: dict, G: dict, W: dict, sign_u: dict, sign_v: dict, spec, group: int, low: int, high: int,
                   budget: float, block: int = 128, lam: float = 0.01) -> dict:
    """A transformer block: scores, the W2 -> W3 allocation, then each sublayer through
    Algorithms 1 and 2 at its allocated bit width."""
    sc = block_scores(X, G, W, spec)
    params = {name: d_out * d_in for name, _, d_out, d_in in spec}
    bits = allocate_bits({n: sc[n]["s_post"] for n, _, _, _ in spec}, params, low, high, budget)
    res = {}
    for name, grp, _, _ in spec:
        res[name] = pipeline(X[grp], G[name], W[name], sign_u[name], sign_v[name], bits[name], group, block, lam)
    return {"scores": sc, "bits": bits, "layers": res}


# ----------------------------------------------------------------------------------
# Inference with the quantized layer (Algorithm 2's revert; Sec. 3.2: the scales are
# reverted elementwise and U, V applied to activations at inference).
# ----------------------------------------------------------------------------------
def infer(codes, scale, zero, group: int, s_x, s_g, sign_u, sign_v, x) -> np.ndarray:
    """y = W^ x^T for tokens x [B, d_in] (returned [B, d_out]), W^ the dense reverted
    weight S_G^-1 U^T Q' V S_X^-1 in float64."""
    d_out, d_in = np.asarray(codes).shape
    U = rht_matrix(d_out, sign_u)
    V = rht_matrix(d_in, sign_v)
    What = revert(dequant(codes, np.asarray(scale, np.float64), np.asarray(zero, np.float64), group),
                  np.asarray(s_x, np.float64), np.asarray(s_g, np.float64), U, V)
    return np.asarray(x, np.float64) @ What.T


# ----------------------------------------------------------------------------------
# BiIP statistics (Prop. 2; Sec. 3.2 "CV_in / CV_out"; the appendix on weight distributions).
# ----------------------------------------------------------------------------------
def biip_scales_exp(W, hx, hg, ex: float, eg: float):
    """Eq. (rescale) with the exponent as a parameter: s_x = (h_x / a)^ex, s_g = (h_g / r)^eg
    (ex = eg = 1/4 is the paper's; Prop. 2's sweep varies it). Dead channels get 1."""
    W = np.asarray(W, dtype=np.float64)
    a = np.sum(W * W, axis=0)
    r = np.sum(W * W, axis=1)
    hx = np.asarray(hx, np.float64)
    hg = np.asarray(hg, np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        sx = np.where((hx > 0) & (a > 0), (hx / a) ** ex, 1.0)
        sg = np.where((hg > 0) & (r > 0), (hg / r) ** eg, 1.0)
    return sx, sg


def norm_cv(W) -> tuple:
    """(CV_in, CV_out): coefficient of variation (population standard deviation over mean)
    of the column norms ||W[:, j]|| and of the row norms ||W[i, :]||."""
    W = np.asarray(W, dtype=np.float64)
    c = np.sqrt(np.sum(W * W, axis=0))
    r = np.sqrt(np.sum(W * W, axis=1))
    return float(np.std(c) / np.mean(c)), float(np.std(r) / np.mean(r))


def rho(h, a) -> float:
    """Prop. 2's gain of the rescale over none: (sum sqrt(h a))^2 / (sum h sum a) <= 1."""
    h = np.asarray(h, np.float64)
    a = np.asarray(a, np.float64)
    return float(np.sum(np.sqrt(h * a)) ** 2 / (np.sum(h) * np.sum(a)))


def prop2_bound(h, a, s) -> float:
    """The rescale-dependent factor of Prop. 2's expected loss: (sum h / s^2)(sum s^2 a)."""
    h = np.asarray(h, np.float64)
    a = np.asarray(a, np.float64)
    s = np.asarray(s, np.float64)
    return float(np.sum(h / s ** 2) * np.sum(s ** 2 * a))
