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
