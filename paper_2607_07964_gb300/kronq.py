"""Thin Python binding of libkronq (include/kronq.h): the same entry points, taking torch
CUDA tensors. It only checks and marshals arguments (pointers, sizes, the current CUDA
stream); every step of the computation runs in the library's kernels. There is no CPU
or PyTorch fallback: if libkronq.so is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
# KQ_DEBUG=1 selects the debug build (bounds checks before the kernels' stores; see
# kq_debug_status), built with `python -m paper_2607_07964_gb300.build --debug`
LIB_PATH = os.path.join(_HERE, "libkronq_debug.so" if os.environ.get("KQ_DEBUG") == "1" else "libkronq.so")

KQ_OK, KQ_ERR_INVALID_ARG, KQ_ERR_UNSUPPORTED, KQ_ERR_NOT_PD = 0, 1, 2, 3
KQ_ERR_CUDA, KQ_ERR_TIMEOUT, KQ_ERR_WORKSPACE, KQ_ERR_NONFINITE = 4, 5, 6, 7
KQ_FWD, KQ_INV, KQ_FWD_SYM = 0, 1, 2
KQ_TRAIL_FP32, KQ_TRAIL_3XTF32 = 0, 1
KQ_SYRK_CHUNK_TOKENS = 512

_lib = None


class KronqError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: {status_name(status)} ({msg})")
        self.status = status


def lib() -> ctypes.CDLL:
    """Load libkronq.so (built by paper_2607_07964_gb300.build); raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2607_07964_gb300.build` (needs nvcc)")
        L = ctypes.CDLL(LIB_PATH)
        P, I64, I, F, SZ = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
        sig = {
            "kq_last_error": ([], ctypes.c_char_p),
            "kq_status_name": ([I], ctypes.c_char_p),
            "kq_version": ([], I),
            "kq_launch_count": ([], ctypes.c_uint64),
            "kq_graph_instantiate": ([P, I, P], I),
            "kq_graph_launch": ([P, P], I),
            "kq_graph_exec_destroy": ([P], I),
            "kq_check": ([P, I, P, P], I),
            "kq_selftest_timeout": ([P, I64, P], I),
            "kq_debug_build": ([], I),
            "kq_debug_status": ([P, P, I], I),
            "kq_selftest_bounds": ([P, I64, P], I),
            "kq_selftest_div": ([P, P, I64, P, P], I),
            "kq_accum_factor": ([P, I64, I64, I64, P, I, P, P, P], I),
            "kq_compute_scales": ([P, I64, I64, P, P, P, P, P], I),
            "kq_compute_scales_diag": ([P, I64, I64, P, P, P, P, P], I),
            "kq_compute_scales_exp": ([P, I64, I64, P, P, P, P, F, F, P], I),
            "kq_biip_stats_workspace": ([I64, I64], SZ),
            "kq_biip_stats": ([P, I64, I64, P, P, P, P, SZ, P], I),
            "kq_traces_diag": ([P, P, I64, P, P, I64, P, P], I),
            "kq_factor_diag_workspace": ([I64, I64], SZ),
            "kq_factor_diag": ([P, I64, I64, I64, P, P, P, SZ, P], I),
            "kq_traces": ([P, P, I64, P, P, I64, P, P], I),
            "kq_rotate_in": ([P, I64, I64, P, P, P, I, P], I),
            "kq_rotate_out": ([P, I64, I64, P, P, P, I, P], I),
            "kq_chol_inv_workspace": ([I64], SZ),
            "kq_chol_inv": ([P, I64, F, P, P, P, SZ, P], I),
            "kq_chol_inv_noalloc": ([P, I64, F, P, P, P], I),
            "kq_obs_quantize_workspace": ([I64, I64, I, I, I], SZ),
            "kq_obs_quantize": ([P, I64, I64, P, P, I, I, I, I, P, P, P, P, P, P, P, SZ, P], I),
            "kq_accum_drift_workspace": ([I64, I64], SZ),
            "kq_accum_drift": ([P, P, I64, I64, I64, P, I, P, P, SZ, P], I),
            "kq_packed_codes_bytes": ([I64, I64, I], SZ),
            "kq_pack_codes": ([P, I64, I64, I, P, P], I),
            "kq_infer_workspace": ([I64, I64, I64], SZ),
            "kq_infer": ([P, P, P, I64, I64, I, I, P, P, P, P, P, I64, P, P, P, SZ, P], I),
            "kq_gptaq_p_workspace": ([I64], SZ),
            "kq_gptaq_p": ([P, P, I64, F, P, P, P, SZ, P], I),
            "kq_dequant_revert": ([P, P, P, I64, I64, I, P, P, P, P, P, P], I),
            "kq_proxy_loss_workspace": ([I64, I64], SZ),
            "kq_proxy_loss": ([P, P, I64, I64, P, P, P, P, SZ, P], I),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def status_name(s: int) -> str:
    return lib().kq_status_name(int(s)).decode()


def last_error() -> str:
    return lib().kq_last_error().decode()


def _ok(st: int, where: str) -> None:
    if st != KQ_OK:
        raise KronqError(st, where, last_error())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, name, dtype, shape=None, contiguous=True):
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if contiguous and not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def version() -> int:
    return lib().kq_version()


def launch_count() -> int:
    """Kernels launched by libkronq so far in this process."""
    return int(lib().kq_launch_count())


def kq_check(info=None, reset: bool = True, stream=None) -> tuple[int, int]:
    """Synchronize the stream and read the device error word; returns (status, raw)."""
    raw = ctypes.c_int(0)
    st = lib().kq_check(_ptr(info), int(reset), ctypes.byref(raw), _stream(stream))
    return st, raw.value


def kq_debug_build() -> bool:
    return bool(lib().kq_debug_build())


DEBUG_UNITS = ("api", "syrk", "biip", "chol", "obs", "trail_tc", "gptaq", "infer", "check")


def kq_debug_status(reset: bool = True) -> tuple[str | None, int]:
    """(source file, line) of the first failed bounds check of the debug build, or (None, 0)."""
    unit, line = ctypes.c_int(-1), ctypes.c_int(0)
    _ok(lib().kq_debug_status(ctypes.byref(unit), ctypes.byref(line), int(reset)), "kq_debug_status")
    return (DEBUG_UNITS[unit.value] if unit.value >= 0 else None), line.value


def kq_selftest_bounds(buf, n: int, stream=None) -> None:
    """buf: n + 1 float32 on the device; writes buf[i] = i for i <= n under a check against n."""
    _need(buf, "buf", torch.float32, (n + 1,))
    _ok(lib().kq_selftest_bounds(_ptr(buf), int(n), _stream(stream)), "kq_selftest_bounds")


def kq_selftest_timeout(info, limit_us: int, stream=None) -> None:
    """A kernel whose bounded wait runs out (nothing arrives); *info gets -KQ_ERR_TIMEOUT."""
    _need(info, "info", torch.int32)
    _ok(lib().kq_selftest_timeout(_ptr(info), int(limit_us), _stream(stream)), "kq_selftest_timeout")


def kq_graph_instantiate(graph: int, use_node_priority: bool = True) -> int:
    """cudaGraphExec_t (as an int) for the cudaGraph_t `graph`, honouring the captured
    per-node priorities when use_node_priority."""
    ex = ctypes.c_void_p()
    _ok(lib().kq_graph_instantiate(ctypes.c_void_p(graph), int(use_node_priority), ctypes.byref(ex)),
        "kq_graph_instantiate")
    return int(ex.value)


def kq_graph_launch(exec_: int, stream=None) -> None:
    _ok(lib().kq_graph_launch(ctypes.c_void_p(exec_), _stream(stream)), "kq_graph_launch")


def kq_graph_exec_destroy(exec_: int) -> None:
    _ok(lib().kq_graph_exec_destroy(ctypes.c_void_p(exec_)), "kq_graph_exec_destroy")


def kq_selftest_div(a, b, mismatches, stream=None) -> None:
    """mismatches (+)= the count of a[i] / b[i] where the sweep's division differs from IEEE
    round-to-nearest division in any bit; a, b fp32 of one shape, mismatches one int64."""
    _need(a, "a", torch.float32)
    _need(b, "b", torch.float32, tuple(a.shape))
    _need(mismatches, "mismatches", torch.int64, (1,))
    _ok(lib().kq_selftest_div(_ptr(a), _ptr(b), a.numel(), _ptr(mismatches), _stream(stream)), "kq_selftest_div")


def kq_accum_factor(A, H, accumulate: bool = False, trace=None, info=None, stream=None) -> None:
    """H (+)= A^T A; A [T, d] bf16 (row stride may exceed d), H [d, d] fp32."""
    if A.dim() != 2 or A.stride(1) != 1:
        raise ValueError("A must be 2-D with unit column stride")
    T, d = A.shape
    _need(A, "A", torch.bfloat16, contiguous=False)
    _need(H, "H", torch.float32, (d, d))
    _need(trace, "trace", torch.float64)
    _need(info, "info", torch.int32)
    _ok(lib().kq_accum_factor(_ptr(A), T, d, A.stride(0), _ptr(H), int(accumulate), _ptr(trace),
                              _ptr(info), _stream(stream)), "kq_accum_factor")


def kq_accum_drift_workspace(T: int, d: int) -> int:
    """Bytes for one pass over all T tokens (a smaller workspace makes token chunks)."""
    return int(lib().kq_accum_drift_workspace(T, d))


def kq_accum_drift(Xt, X, D, accumulate: bool = False, info=None, ws=None, stream=None) -> None:
    """D (+)= (X~ - X)^T X; Xt (X~) and X [T, d] bf16 with the same row stride, D [d, d] fp32."""
    if X.dim() != 2 or X.stride(1) != 1 or Xt.shape != X.shape or Xt.stride() != X.stride():
        raise ValueError("X~ and X must be 2-D, same shape and strides, unit column stride")
    T, d = X.shape
    _need(Xt, "Xt", torch.bfloat16, contiguous=False)
    _need(X, "X", torch.bfloat16, contiguous=False)
    _need(D, "D", torch.float32, (d, d))
    _need(info, "info", torch.int32)
    _need(ws, "ws", torch.uint8)
    _ok(lib().kq_accum_drift(_ptr(Xt), _ptr(X), T, d, X.stride(0), _ptr(D), int(accumulate), _ptr(info),
                             _ptr(ws), 0 if ws is None else ws.numel(), _stream(stream)), "kq_accum_drift")


def kq_gptaq_p_workspace(n: int) -> int:
    return int(lib().kq_gptaq_p_workspace(n))


def kq_gptaq_p(Dp, Lt, alpha: float, Pt, ws, info=None, stream=None) -> None:
    """Pt = P^T with P = alpha ((D' L) o M_U) L^T (Proposition 1, Algorithm 2)."""
    n = Lt.shape[0]
    _need(Dp, "Dp", torch.float32, (n, n))
    _need(Lt, "Lt", torch.float32, (n, n))
    _need(Pt, "Pt", torch.float32, (n, n))
    _need(ws, "ws", torch.uint8)
    _need(info, "info", torch.int32)
    _ok(lib().kq_gptaq_p(_ptr(Dp), _ptr(Lt), n, float(alpha), _ptr(Pt), _ptr(info), _ptr(ws),
                         0 if ws is None else ws.numel(), _stream(stream)), "kq_gptaq_p")


def kq_compute_scales(W, H_X, H_G, s_x, s_g, stream=None) -> None:
    """s_x and/or s_g (each side computed only if its output is given)."""
    d_out, d_in = W.shape
    _need(W, "W", torch.float32)
    _need(H_X, "H_X", torch.float32, (d_in, d_in))
    _need(H_G, "H_G", torch.float32, (d_out, d_out))
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _ok(lib().kq_compute_scales(_ptr(W), d_out, d_in, _ptr(H_X), _ptr(H_G), _ptr(s_x), _ptr(s_g),
                                _stream(stream)), "kq_compute_scales")


def kq_compute_scales_exp(W, H_X, H_G, s_x, s_g, ex: float, eg: float, stream=None) -> None:
    """Scales with the exponent as a parameter (1/4: kq_compute_scales)."""
    d_out, d_in = W.shape
    _need(W, "W", torch.float32)
    _need(H_X, "H_X", torch.float32, (d_in, d_in))
    _need(H_G, "H_G", torch.float32, (d_out, d_out))
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _ok(lib().kq_compute_scales_exp(_ptr(W), d_out, d_in, _ptr(H_X), _ptr(H_G), _ptr(s_x), _ptr(s_g), float(ex),
                                    float(eg), _stream(stream)), "kq_compute_scales_exp")


def kq_biip_stats_workspace(d_out: int, d_in: int) -> int:
    return int(lib().kq_biip_stats_workspace(d_out, d_in))


def kq_biip_stats(W, H_X, H_G, out, ws, stream=None) -> None:
    """out [4] float64 = [CV_in, CV_out, rho_in, rho_out] of W with the factors' diagonals."""
    d_out, d_in = W.shape
    _need(W, "W", torch.float32)
    _need(H_X, "H_X", torch.float32, (d_in, d_in))
    _need(H_G, "H_G", torch.float32, (d_out, d_out))
    _need(out, "out", torch.float64, (4,))
    _need(ws, "ws", torch.uint8)
    _ok(lib().kq_biip_stats(_ptr(W), d_out, d_in, _ptr(H_X), _ptr(H_G), _ptr(out), _ptr(ws),
                            0 if ws is None else ws.numel(), _stream(stream)), "kq_biip_stats")


def kq_traces(H_X, s_x, H_G, s_g, out, stream=None) -> None:
    """Sensitivity traces; either factor may be None (that side of `out` is kept)."""
    d_in = 0 if H_X is None else H_X.shape[0]
    d_out = 0 if H_G is None else H_G.shape[0]
    _need(H_X, "H_X", torch.float32, (d_in, d_in))
    _need(H_G, "H_G", torch.float32, (d_out, d_out))
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _need(out, "out", torch.float64, (6,))
    _ok(lib().kq_traces(_ptr(H_X), _ptr(s_x), d_in, _ptr(H_G), _ptr(s_g), d_out, _ptr(out),
                        _stream(stream)), "kq_traces")


def kq_factor_diag_workspace(T: int, d: int) -> int:
    return int(lib().kq_factor_diag_workspace(T, d))


def kq_factor_diag(A, diag, trace=None, ws=None, stream=None) -> None:
    """diag(A^T A) (fp64 sums, fp32 result) and optionally its total; A [T, d] bf16."""
    if A.dim() != 2 or A.stride(1) != 1:
        raise ValueError("A must be 2-D with unit column stride")
    T, d = A.shape
    _need(A, "A", torch.bfloat16, contiguous=False)
    _need(diag, "diag", torch.float32, (d,))
    _need(trace, "trace", torch.float64)
    _need(ws, "ws", torch.uint8)
    _ok(lib().kq_factor_diag(_ptr(A), T, d, A.stride(0), _ptr(diag), _ptr(trace), _ptr(ws),
                             0 if ws is None else ws.numel(), _stream(stream)), "kq_factor_diag")


def kq_compute_scales_diag(W, hx_diag, hg_diag, s_x, s_g, stream=None) -> None:
    d_out, d_in = W.shape
    _need(W, "W", torch.float32)
    _need(hx_diag, "hx_diag", torch.float32, (d_in,))
    _need(hg_diag, "hg_diag", torch.float32, (d_out,))
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _ok(lib().kq_compute_scales_diag(_ptr(W), d_out, d_in, _ptr(hx_diag), _ptr(hg_diag), _ptr(s_x), _ptr(s_g),
                                     _stream(stream)), "kq_compute_scales_diag")


def kq_traces_diag(hx_diag, s_x, hg_diag, s_g, out, stream=None) -> None:
    d_in = 0 if hx_diag is None else hx_diag.shape[0]
    d_out = 0 if hg_diag is None else hg_diag.shape[0]
    _need(hx_diag, "hx_diag", torch.float32, (d_in,))
    _need(hg_diag, "hg_diag", torch.float32, (d_out,))
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _need(out, "out", torch.float64, (6,))
    _ok(lib().kq_traces_diag(_ptr(hx_diag), _ptr(s_x), d_in, _ptr(hg_diag), _ptr(s_g), d_out, _ptr(out),
                             _stream(stream)), "kq_traces_diag")


def kq_rotate_in(W, H_X, s_x, sign_v, direction: int = KQ_FWD, stream=None, d_out: int = 0) -> None:
    """W may be None (then only H_X is transformed, forward direction)."""
    if W is not None:
        d_out, d_in = W.shape
    else:
        d_in = H_X.shape[0]
    _need(W, "W", torch.float32)
    _need(H_X, "H_X", torch.float32, (d_in, d_in))
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(sign_v, "sign_v", torch.int8, (d_in,))
    _ok(lib().kq_rotate_in(_ptr(W), d_out, d_in, _ptr(H_X), _ptr(s_x), _ptr(sign_v), int(direction),
                           _stream(stream)), "kq_rotate_in")


def kq_rotate_out(W, H_G, s_g, sign_u, direction: int = KQ_FWD, stream=None, d_in: int = 0) -> None:
    """W may be None (then only H_G is transformed, forward direction)."""
    if W is not None:
        d_out, d_in = W.shape
    else:
        d_out = H_G.shape[0]
    _need(W, "W", torch.float32)
    _need(H_G, "H_G", torch.float32, (d_out, d_out))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _need(sign_u, "sign_u", torch.int8, (d_out,))
    _ok(lib().kq_rotate_out(_ptr(W), d_out, d_in, _ptr(H_G), _ptr(s_g), _ptr(sign_u), int(direction),
                            _stream(stream)), "kq_rotate_out")


def kq_chol_inv_workspace(n: int) -> int:
    return int(lib().kq_chol_inv_workspace(n))


def kq_chol_inv(H, damp_rel: float, Lt, info, ws, stream=None) -> None:
    n = H.shape[0]
    _need(H, "H", torch.float32, (n, n))
    _need(Lt, "Lt", torch.float32, (n, n))
    _need(info, "info", torch.int32)
    _need(ws, "ws", torch.uint8)
    _ok(lib().kq_chol_inv(_ptr(H), n, float(damp_rel), _ptr(Lt), _ptr(info), _ptr(ws),
                          0 if ws is None else ws.numel(), _stream(stream)), "kq_chol_inv")


KQ_CHOL_NOALLOC_MAX_N = 1024


def kq_chol_inv_noalloc(H, damp_rel: float, Lt, info=None, stream=None) -> None:
    """kq_chol_inv without a caller workspace (n <= KQ_CHOL_NOALLOC_MAX_N): the library's
    own fixed device array serves as scratch. Calls must not overlap on the GPU."""
    n = H.shape[0]
    _need(H, "H", torch.float32, (n, n))
    _need(Lt, "Lt", torch.float32, (n, n))
    _need(info, "info", torch.int32)
    _ok(lib().kq_chol_inv_noalloc(_ptr(H), n, float(damp_rel), _ptr(Lt), _ptr(info), _stream(stream)),
        "kq_chol_inv_noalloc")


def kq_obs_quantize_workspace(d_out: int, d_in: int, block: int = 128, mode: int = KQ_TRAIL_FP32,
                              with_p: bool = False) -> int:
    return int(lib().kq_obs_quantize_workspace(d_out, d_in, block, mode, int(with_p)))


def kq_obs_quantize(W, Lt, bits: int, group: int, block: int, codes, scale, zero, col_loss=None,
                    pre_q=None, ws=None, stream=None, mode: int = KQ_TRAIL_FP32, info=None, Pt=None) -> None:
    """mode: KQ_TRAIL_FP32 (fp32-ordered trailing update, bit-exact) or KQ_TRAIL_3XTF32.
    Pt: P^T from kq_gptaq_p for the GPTAQ drift correction, or None (GPTQ mode)."""
    d_out, d_in = W.shape
    ng = 1 if group == 0 else -(-d_in // group)
    _need(W, "W", torch.float32)
    _need(Lt, "Lt", torch.float32, (d_in, d_in))
    _need(Pt, "Pt", torch.float32, (d_in, d_in))
    _need(codes, "codes", torch.uint8, (d_out, d_in))
    _need(scale, "scale", torch.float32, (d_out, ng))
    _need(zero, "zero", torch.int32, (d_out, ng))
    _need(col_loss, "col_loss", torch.float32, (d_in,))
    _need(pre_q, "pre_q", torch.float32, (d_out, d_in))
    _need(ws, "ws", torch.uint8)
    _need(info, "info", torch.int32)
    _ok(lib().kq_obs_quantize(_ptr(W), d_out, d_in, _ptr(Lt), _ptr(Pt), bits, group, block, mode, _ptr(codes),
                              _ptr(scale), _ptr(zero), _ptr(col_loss), _ptr(pre_q), _ptr(info), _ptr(ws),
                              0 if ws is None else ws.numel(), _stream(stream)), "kq_obs_quantize")


def kq_packed_codes_bytes(d_out: int, d_in: int, bits: int) -> int:
    return int(lib().kq_packed_codes_bytes(d_out, d_in, bits))


def kq_pack_codes(codes, bits: int, packed, stream=None) -> None:
    """codes [d_out, d_in] uint8 -> packed words (int32 tensor of kq_packed_codes_bytes / 4)."""
    d_out, d_in = codes.shape
    _need(codes, "codes", torch.uint8)
    _need(packed, "packed", torch.int32, (kq_packed_codes_bytes(d_out, d_in, bits) // 4,))
    _ok(lib().kq_pack_codes(_ptr(codes), d_out, d_in, bits, _ptr(packed), _stream(stream)), "kq_pack_codes")


def kq_infer_workspace(B: int, d_in: int, d_out: int) -> int:
    return int(lib().kq_infer_workspace(B, d_in, d_out))


def kq_infer(packed, scale, zero, d_out: int, d_in: int, bits: int, group: int, s_x, s_g, sign_u, sign_v, x, y,
             ws, stream=None, info=None) -> None:
    """y [B, d_out] = W^ x for x [B, d_in]: the reverted quantized layer applied with online
    Hadamard transforms (Algorithm 2's revert, Sec. 3.2). info: optional int32 device word
    for a timed-out weight stream (read with kq_check)."""
    B = x.shape[0]
    _need(packed, "packed", torch.int32)
    _need(scale, "scale", torch.float32)
    _need(zero, "zero", torch.int32)
    _need(s_x, "s_x", torch.float32, (d_in,))
    _need(s_g, "s_g", torch.float32, (d_out,))
    _need(sign_u, "sign_u", torch.int8, (d_out,))
    _need(sign_v, "sign_v", torch.int8, (d_in,))
    _need(x, "x", torch.float32, (B, d_in))
    _need(y, "y", torch.float32, (B, d_out))
    _need(ws, "ws", torch.uint8)
    _need(info, "info", torch.int32)
    _ok(lib().kq_infer(_ptr(packed), _ptr(scale), _ptr(zero), d_out, d_in, bits, group, _ptr(s_x), _ptr(s_g),
                       _ptr(sign_u), _ptr(sign_v), _ptr(x), B, _ptr(y), _ptr(info), _ptr(ws),
                       0 if ws is None else ws.numel(), _stream(stream)), "kq_infer")


def kq_dequant_revert(codes, scale, zero, group: int, s_x, s_g, sign_u, sign_v, W_hat, stream=None):
    d_out, d_in = codes.shape
    _need(codes, "codes", torch.uint8)
    _need(scale, "scale", torch.float32)
    _need(zero, "zero", torch.int32)
    _need(W_hat, "W_hat", torch.float32, (d_out, d_in))
    _ok(lib().kq_dequant_revert(_ptr(codes), _ptr(scale), _ptr(zero), d_out, d_in, group, _ptr(s_x),
                                _ptr(s_g), _ptr(sign_u), _ptr(sign_v), _ptr(W_hat), _stream(stream)),
        "kq_dequant_revert")


def kq_proxy_loss_workspace(d_out: int, d_in: int) -> int:
    return int(lib().kq_proxy_loss_workspace(d_out, d_in))


def kq_proxy_loss(W, W_hat, H_X, H_G, loss, ws, stream=None) -> None:
    d_out, d_in = W.shape
    _need(W, "W", torch.float32)
    _need(W_hat, "W_hat", torch.float32, (d_out, d_in))
    _need(H_X, "H_X", torch.float32, (d_in, d_in))
    _need(H_G, "H_G", torch.float32, (d_out, d_out))
    _need(loss, "loss", torch.float64, (1,))
    _need(ws, "ws", torch.uint8)
    _ok(lib().kq_proxy_loss(_ptr(W), _ptr(W_hat), d_out, d_in, _ptr(H_X), _ptr(H_G), _ptr(loss),
                            _ptr(ws), ws.numel(), _stream(stream)), "kq_proxy_loss")
