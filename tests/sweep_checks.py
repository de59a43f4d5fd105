"""Checks of the tensor-core (3xTF32) sweep against the oracle, shared by the GPU tests.

The fast mode sums the lazy trailing update in another order than the fp32-ordered
definition, so a code can flip at a rounding tie and the rest of that row then follows
another (equally valid) path. It is judged in two ways:
  * teacher forced, on every checked row (oracle.teacher_forced): the GPU's codes are the
    exact float32 quantization of its own pre-quantization values on its own grids; those
    values are within float32 rounding (2e-5 of |W'_j| + sum_k |E_k R_kj|) of what
    Algorithm 2 computes from the GPU's own earlier errors; its group grids come from the
    block-start values that the same replay gives;
  * against the fp32-ordered oracle sweep: the first difference in each row sits within 1e-4
    quantization steps of a rounding tie, and such first differences are at most 0.1 % of
    the codes compared up to them. After a row's first difference its error feedback takes
    the other (equally valid) path, so later codes of that row differ too; how many depends
    on where the tie falls and on the row length (a flip near the start of a 28672-wide row
    makes most of that row differ), which is why the rate is taken over the independent
    disagreements and the rest of the row is held to the teacher-forced check instead.
"""
import numpy as np

from oracle import kronq_oracle as ref
from oracle import obs_sweep_fp32

# float32 rounding of the update, relative to the magnitudes summed into each value
TF_REL = 2e-5


def check_teacher_forced(Wp, Lt, g, bits, group, block=128, Pt=None, rows=None):
    """g: the GPU's codes, scale, zero, pre_q (host arrays, all rows). rows: the rows to
    replay (all if None)."""
    sel = slice(None) if rows is None else np.asarray(rows)
    codes, scale, zero, pre_q = g["codes"][sel], g["scale"][sel], g["zero"][sel], g["pre_q"][sel]
    tf = ref.teacher_forced(np.asarray(Wp)[sel], Lt, pre_q, codes, scale, zero, bits, group, block, Pt=Pt)
    # (i) codes are the float32 quantization of the GPU's own values, bit for bit
    bad = np.argwhere(tf["codes"] != codes)
    assert bad.size == 0, f"codes differ from quant(pre_q) at {bad[:5].tolist()}"
    # (ii) the values follow Algorithm 2 from the GPU's own errors
    dev = np.abs(pre_q.astype(np.float64) - tf["pre_q"]) / tf["absum"]
    worst = np.unravel_index(int(np.argmax(dev)), dev.shape)
    assert dev[worst] <= TF_REL, (dev[worst], worst)
    # (iii) group grids from the block-start values
    if group:
        maxq = 2 ** bits - 1
        n = Wp.shape[1]
        for gi in range(scale.shape[1]):
            c0, c1 = gi * group, min(n, (gi + 1) * group)
            s_ref, z_ref = ref.quant_params(tf["block_start"][:, c0:c1], bits)
            tol = 2 * TF_REL * tf["absum"][:, c0:c1].max(axis=1) / maxq + 2.0 ** -22 * s_ref
            assert np.all(np.abs(scale[:, gi] - s_ref) <= tol), gi
            assert np.all(np.abs(zero[:, gi] - z_ref) <= 1), gi
            xmin = np.minimum(tf["block_start"][:, c0:c1].min(axis=1), 0.0)
            t = -xmin / s_ref
            off_tie = np.abs((t - np.floor(t)) - 0.5) > 1e-3
            assert np.all((zero[:, gi] == z_ref)[off_tie]), gi
    return tf


def check_against_fp32_sweep(Wp, Lt, g, bits, group, block=128, Pt=None, rows=None, max_rate=1e-3):
    """Each row's first difference from the fp32-ordered sweep is at a rounding tie of the
    oracle's value, and first differences are <= max_rate of the codes compared up to them
    (module docstring). Returns the oracle's sweep and the mismatch mask."""
    sel = slice(None) if rows is None else np.asarray(rows)
    c = obs_sweep_fp32(Wp, Lt, bits, group, block, rows=rows, want_pre_q=True, Pt=Pt)
    codes = g["codes"][sel]
    mis = codes != c["codes"]
    n = codes.shape[1]
    firsts, compared = 0, 0
    for r in range(codes.shape[0]):
        if not mis[r].any():
            compared += n
            continue
        j = int(np.argmax(mis[r]))
        firsts += 1
        compared += j + 1
        gi = 0 if group == 0 else j // group
        x = np.float64(c["pre_q"][r, j]) / np.float64(c["scale"][r, gi])
        assert abs((x - np.floor(x)) - 0.5) <= 1e-4, (r, j)
    assert firsts <= max_rate * compared, (firsts, compared, float(mis.mean()))
    return c, mis


def check_fast_sweep(Wp, Lt, g, bits, group, block=128, Pt=None, rows=None):
    check_teacher_forced(Wp, Lt, g, bits, group, block, Pt=Pt, rows=rows)
    return check_against_fp32_sweep(Wp, Lt, g, bits, group, block, Pt=Pt, rows=rows)
