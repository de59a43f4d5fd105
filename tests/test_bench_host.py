"""Host-side arithmetic of bench.py's CPU-oracle estimate (no GPU)."""
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def test_two_point_line_through_both_samples():
    # 2 s fixed + 1 ms per token: 2.5 s at 500 tokens, 3 s at 1000 -> 2 + 262.144 s
    assert bench.two_point_tokens(2.5, 3.0, 500, 262144) == pytest.approx(2.0 + 262.144)


def test_two_point_without_a_usable_slope_scales_the_larger_sample():
    # the second sample not slower than the first: no negative or zero extrapolation
    assert bench.two_point_tokens(5.0, 4.0, 2048, 262144) == pytest.approx(4.0 * 262144 / 4096)
    assert bench.two_point_tokens(4.0, 4.0, 2048, 262144) == pytest.approx(4.0 * 262144 / 4096)
    assert bench.two_point_tokens(9.0, 1.0, 2048, 262144) > 0


# ---------------------------------------------------------------- host path chunk plan
def _plan(x_tokens, g_tokens, which, T):
    import types
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    return LayerPipeline._chunks(types.SimpleNamespace(chunk_tokens={"X": x_tokens, "G": g_tokens}), which, T)


@pytest.mark.parametrize("which", ["X", "G"])
@pytest.mark.parametrize("chunk", [0, 1, 512, 32768])
@pytest.mark.parametrize("T", [1, 3, 4096, 32768, 100000, 262144])
def test_token_chunks_tile_the_tokens(which, chunk, T):
    """The factor chunks (Alg. 1's online statistic, one accumulate call per chunk) cover
    [0, T) in order, contiguous and non-empty; X's first and G's last chunk of several come
    in quarters."""
    ch = _plan(chunk, chunk, which, T)
    assert ch[0][0] == 0 and ch[-1][1] == T
    assert all(a < b for a, b in ch)
    assert all(ch[i][1] == ch[i + 1][0] for i in range(len(ch) - 1))
    if chunk == 0 or T <= chunk:
        assert ch == [(0, T)]
        return
    full = [(t0, min(T, t0 + chunk)) for t0 in range(0, T, chunk)]
    split = full[0] if which == "X" else full[-1]
    q = -(-(split[1] - split[0]) // 4)
    pieces = [(a, min(split[1], a + q)) for a in range(split[0], split[1], q)]
    assert ch == (pieces + full[1:] if which == "X" else full[:-1] + pieces)
