"""The allocation-free Cholesky entry point (kq_chol_inv_noalloc) against the ordinary
one (kq_chol_inv with a caller workspace).

kq_chol_inv_noalloc serves callers that may not allocate device memory at call time (a
plugin inside a runtime that owns all device memory, or a loop where cudaMalloc would
synchronize): it takes only inputs and outputs and uses a fixed device array owned by the
library. This file is collected last so that a failure here leaves every other test run.
"""
import ctypes

import numpy as np
import pytest
import torch

import kqsynth

pytestmark = pytest.mark.gpu


def test_chol_inv_noalloc_matches_workspace_entry_point():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    from paper_2607_07964_gb300 import kronq as K
    build.build()
    lib = K.lib()
    f = lib.kq_chol_inv_noalloc
    P = ctypes.c_void_p
    f.argtypes = [P, ctypes.c_int64, ctypes.c_float, P, P, P]
    f.restype = ctypes.c_int
    stream = P(torch.cuda.current_stream().cuda_stream)
    # two calls in a row, the second smaller than the first, so it runs on an array that
    # still holds the first call's data
    for n, seed in [(1000, 11), (300, 12)]:
        H = torch.from_numpy(kqsynth.random_spd(n, seed=seed, cond_decay=1.0).astype(np.float32)).cuda()
        info_a = torch.zeros(1, dtype=torch.int32, device="cuda")
        info_b = torch.zeros(1, dtype=torch.int32, device="cuda")
        Lt_a = torch.full((n, n), float("nan"), device="cuda")
        Lt_b = torch.full((n, n), float("nan"), device="cuda")
        ws = torch.empty(K.kq_chol_inv_workspace(n), dtype=torch.uint8, device="cuda")
        K.kq_chol_inv(H, 0.01, Lt_a, info_a, ws)
        st = f(P(H.data_ptr()), n, 0.01, P(Lt_b.data_ptr()), P(info_b.data_ptr()), stream)
        assert st == K.KQ_OK, K.last_error()
        assert K.kq_check(info_a)[0] == K.KQ_OK
        assert K.kq_check(info_b)[0] == K.KQ_OK
        # the same kernels on the same stream with the same scratch layout: the same bits,
        # so any byte read from the previous call's contents would show
        assert torch.isfinite(Lt_b).all()
        assert torch.equal(Lt_a, Lt_b)


def test_chol_inv_noalloc_rejects_oversize():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import kronq as K
    n = K.KQ_CHOL_NOALLOC_MAX_N + 1
    H = torch.zeros((n, n), device="cuda")
    Lt = torch.zeros((n, n), device="cuda")
    with pytest.raises(K.KronqError) as e:
        K.kq_chol_inv_noalloc(H, 0.01, Lt)
    assert e.value.status == K.KQ_ERR_WORKSPACE
    assert "1024" in str(e.value)
