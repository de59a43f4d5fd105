"""Host-side checks of the C ABI that need no GPU: the library builds and loads, exports
every entry point include/kronq.h declares, and rejects bad arguments on the host before
touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kronq.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_07964_gb300 import build, kronq
    build.build()
    return kronq.lib()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"KQ_API\s+[\w\s\*]+?\b(kq_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for required in ["kq_accum_factor", "kq_compute_scales", "kq_rotate_in", "kq_rotate_out",
                     "kq_chol_inv", "kq_obs_quantize", "kq_traces", "kq_check", "kq_accum_drift",
                     "kq_gptaq_p"]:
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_status_names_and_version(lib):
    from paper_2607_07964_gb300 import kronq
    assert kronq.status_name(0) == "KQ_OK"
    assert kronq.status_name(3) == "KQ_ERR_NOT_PD"
    assert kronq.version() >= 100


def test_workspace_queries(lib):
    from paper_2607_07964_gb300 import kronq
    assert kronq.kq_chol_inv_workspace(256) >= 2 * 256 * 256 * 4
    assert kronq.kq_chol_inv_workspace(200) >= 2 * 256 * 256 * 4   # padded to the block size
    assert kronq.kq_chol_inv_workspace(0) == 0
    assert kronq.kq_obs_quantize_workspace(64, 256, 128) >= 64 * 256 * 4
    assert kronq.kq_obs_quantize_workspace(64, 256, 128, kronq.KQ_TRAIL_3XTF32) >= 3 * 64 * 256 * 4 + 2 * 256 * 256 * 4
    assert kronq.kq_obs_quantize_workspace(64, 256, 128, 5) == 0
    # with P: packed P blocks and -Wpre (fp32), or its split and the split P (tensor cores)
    assert (kronq.kq_obs_quantize_workspace(64, 256, 128, kronq.KQ_TRAIL_FP32, True) >=
            kronq.kq_obs_quantize_workspace(64, 256, 128) + 2 * 128 * 128 * 4 + 64 * 256 * 4)
    assert (kronq.kq_obs_quantize_workspace(64, 256, 128, kronq.KQ_TRAIL_3XTF32, True) >=
            kronq.kq_obs_quantize_workspace(64, 256, 128, kronq.KQ_TRAIL_3XTF32) + 2 * 128 * 128 * 4
            + 2 * 64 * 256 * 4 + 2 * 256 * 256 * 4)
    assert kronq.kq_proxy_loss_workspace(8, 8) >= 3 * 64 * 4
    assert kronq.kq_accum_drift_workspace(100, 64) == 2 * 128 * 64 * 2   # tokens padded to 64
    assert kronq.kq_accum_drift_workspace(0, 64) == 0
    assert kronq.kq_gptaq_p_workspace(256) >= 6 * 256 * 256 * 4


def test_host_side_argument_errors(lib):
    """Calls with invalid arguments return before any CUDA call (safe without a GPU)."""
    from paper_2607_07964_gb300 import kronq as K
    P = ctypes.c_void_p
    fake = P(256)   # never dereferenced: validation fails first
    assert lib.kq_accum_factor(None, 16, 8, 8, None, 0, None, None, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_accum_factor(fake, 16, 8, 4, fake, 0, None, None, None) == K.KQ_ERR_INVALID_ARG  # lda < d
    assert lib.kq_accum_factor(P(258), 16, 8, 8, fake, 0, None, None, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_chol_inv(None, 8, 0.01, None, None, None, 0, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_chol_inv(fake, 8, 0.01, fake, None, None, 0, None) == K.KQ_ERR_WORKSPACE
    assert lib.kq_chol_inv(fake, 8, -1.0, fake, None, fake, 1 << 20, None) == K.KQ_ERR_INVALID_ARG
    # rotation sizes without a Hadamard construction
    assert lib.kq_rotate_in(fake, 4, 100, None, None, fake, 0, None) == K.KQ_ERR_UNSUPPORTED
    assert lib.kq_rotate_out(fake, 100, 4, None, None, fake, 0, None) == K.KQ_ERR_UNSUPPORTED
    assert lib.kq_rotate_in(fake, 4, 28 * 2048, None, None, fake, 0, None) == K.KQ_ERR_UNSUPPORTED
    # sweep: block must be 128 and group in {0, block}
    # (W, d_out, d_in, Lt, Pt, bits, group, block, mode, codes, scale, zero, col_loss, pre_q,
    #  info, ws, ws_bytes, stream)
    args = [fake, 4, 256, fake, None, 4, 64, 128, 0, fake, fake, fake, None, None, None, fake, 1 << 30, None]
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_UNSUPPORTED
    args[7] = 64
    args[6] = 0
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_UNSUPPORTED
    args[7], args[5] = 128, 9
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_INVALID_ARG
    args[5], args[8] = 4, 7                       # unknown trailing-update mode
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_INVALID_ARG
    args[8], args[2] = K.KQ_TRAIL_3XTF32, 258     # tensor-core mode needs d_in % 4 == 0
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_UNSUPPORTED
    args[8], args[2], args[4] = 0, 264, fake      # the drift correction needs d_in % 16 == 0
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_UNSUPPORTED
    args[2], args[4], args[16] = 256, None, 16
    assert lib.kq_obs_quantize(*args) == K.KQ_ERR_WORKSPACE
    assert "workspace" in K.last_error()
    # drift statistic: X~ and X needed, d % 8 == 0, 16-byte alignment, a workspace
    assert lib.kq_accum_drift(None, fake, 16, 8, 8, fake, 0, None, fake, 1 << 20, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_accum_drift(fake, fake, 16, 12, 16, fake, 0, None, fake, 1 << 20, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_accum_drift(P(264), fake, 16, 8, 8, fake, 0, None, fake, 1 << 20, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_accum_drift(fake, fake, 16, 8, 8, fake, 0, None, None, 0, None) == K.KQ_ERR_WORKSPACE
    assert lib.kq_accum_drift(fake, fake, 16, 8, 8, fake, 0, None, fake, 100, None) == K.KQ_ERR_WORKSPACE
    # correction matrix: n % 4 == 0 and a workspace
    assert lib.kq_gptaq_p(None, fake, 8, 0.25, fake, None, fake, 1 << 20, None) == K.KQ_ERR_INVALID_ARG
    assert lib.kq_gptaq_p(fake, fake, 6, 0.25, fake, None, fake, 1 << 20, None) == K.KQ_ERR_UNSUPPORTED
    assert lib.kq_gptaq_p(fake, fake, 8, 0.25, fake, None, fake, 16, None) == K.KQ_ERR_WORKSPACE
    # inference: B in 1..8, bits in {2, 3, 4, 8}, d_in a multiple of 128
    args = [fake, fake, fake, 64, 256, 4, 128, fake, fake, fake, fake, fake, 9, fake, None, fake, 1 << 20, None]
    assert lib.kq_infer(*args) == K.KQ_ERR_INVALID_ARG
    args[12], args[5] = 1, 5
    assert lib.kq_infer(*args) == K.KQ_ERR_UNSUPPORTED
    args[5], args[4] = 4, 200
    assert lib.kq_infer(*args) == K.KQ_ERR_UNSUPPORTED
    assert lib.kq_pack_codes(fake, 4, 200, 4, fake, None) == K.KQ_ERR_UNSUPPORTED
    assert K.kq_packed_codes_bytes(4, 256, 3) == 4 * 256 // 2 and K.kq_packed_codes_bytes(4, 256, 5) == 0


def test_no_cpu_fallback(monkeypatch):
    """The binding has no CPU path: host tensors are refused before any call, and a missing
    library makes every call raise instead of computing something else."""
    import torch
    from paper_2607_07964_gb300 import kronq as K
    A = torch.zeros((64, 8), dtype=torch.bfloat16)
    H = torch.zeros((8, 8), dtype=torch.float32)
    with pytest.raises(ValueError, match="CUDA tensor"):
        K.kq_accum_factor(A, H)
    monkeypatch.setattr(K, "_lib", None)
    monkeypatch.setattr(K, "LIB_PATH", os.path.join(ROOT, "no_such_dir", "libkronq.so"))
    with pytest.raises(RuntimeError, match="missing"):
        K.lib()
    with pytest.raises(RuntimeError, match="missing"):
        K.kq_chol_inv_workspace(256)
