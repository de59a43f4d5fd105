"""A transformer block's linear sublayers through the KronQ path with the mixed-precision
allocation of Sec. 3.3 (Eq. sensitivity: s = tr(H_G) tr(H_X), computed post-BiIP) and
Sec. 5 ("Results on Mixed-precision": the most sensitive sublayers are upgraded from W2 to
W3 one at a time).

Sublayers that read the same input (q, k, v; gate, up) share one H_X accumulation. The
steps: every factor (one H_X per input, one H_G per sublayer) -> scales and traces per
sublayer -> the allocation (a host decision on the scores) -> each sublayer's rotations,
Cholesky and sweep at its bit width, `lanes` sublayers at a time on their own streams.
Everything runs in libkronq's kernels; this module only orders the calls and makes the
allocation.
"""
from __future__ import annotations

import torch

from . import kronq as kq
from .pipeline import LayerPipeline


def allocate_bits(scores: dict, params: dict, low: int, high: int, budget: float) -> dict:
    """Upgrade sublayers from `low` to `high` bits in descending score while the
    parameter-weighted mean bit width stays within `budget`; the first upgrade that would
    exceed it ends the allocation (ties keep the order of `scores`)."""
    names = list(scores)
    ranked = sorted(names, key=lambda n: (-scores[n], names.index(n)))
    total = sum(params[n] for n in names)
    bits = {n: low for n in names}
    extra = 0
    for n in ranked:
        extra_next = extra + (high - low) * params[n]
        if low + extra_next / total > budget:
            break
        bits[n] = high
        extra = extra_next
    return bits


class BlockQuantizer:
    """Buffers for one block shape. spec: (name, input group, d_out, d_in) per sublayer."""

    def __init__(self, spec, group: int, block: int = 128, damp: float = 0.01, low_bits: int = 2,
                 high_bits: int = 3, budget: float = 2.5, device: str = "cuda", trailing: str = "3xtf32",
                 lanes: int = 2):
        self.spec = list(spec)
        self.low, self.high, self.budget = low_bits, high_bits, budget
        self.lanes = max(1, lanes)
        f32 = dict(dtype=torch.float32, device=device)
        d_in_of = {}
        for name, grp, d_out, d_in in self.spec:
            if d_in_of.setdefault(grp, d_in) != d_in:
                raise ValueError(f"input group {grp} has two widths")
        self.groups = list(d_in_of)
        self.HX = {g: torch.empty((d, d), **f32) for g, d in d_in_of.items()}
        self.HG = {name: torch.empty((d_out, d_out), **f32) for name, _, d_out, _ in self.spec}
        self.info = torch.zeros((1,), dtype=torch.int32, device=device)
        self.pipes = {name: LayerPipeline(d_out, d_in, low_bits, group, block, damp, device=device,
                                          want_col_loss=False, trailing=trailing, g_chunk_tokens=0)
                      for name, _, d_out, d_in in self.spec}
        self.lane_streams = [torch.cuda.Stream(device=device) for _ in range(self.lanes)]
        self.params = {name: d_out * d_in for name, _, d_out, d_in in self.spec}

    def factors(self, X: dict, G: dict, stream) -> None:
        """Alg. 1's statistics: one H_X per input (shared by its sublayers), one H_G per
        sublayer."""
        for g in self.groups:
            kq.kq_accum_factor(X[g], self.HX[g], info=self.info, stream=stream)
        for name, _, _, _ in self.spec:
            kq.kq_accum_factor(G[name], self.HG[name], info=self.info, stream=stream)

    def scores(self, W: dict, stream) -> dict:
        """S_X, S_G (Eq. rescale) and the raw and post-BiIP traces of every sublayer, into its
        pipeline's buffers; returns {name: (trHX, trHG, s, trHX', trHG', s')} on the host."""
        for name, grp, _, _ in self.spec:
            p = self.pipes[name]
            kq.kq_compute_scales(W[name], self.HX[grp], self.HG[name], p.s_x, p.s_g, stream=stream)
            kq.kq_traces(self.HX[grp], p.s_x, self.HG[name], p.s_g, p.traces, stream=stream)
        tr = torch.stack([self.pipes[name].traces for name, _, _, _ in self.spec]).cpu()   # synchronizes
        return {name: tuple(float(v) for v in tr[i]) for i, (name, _, _, _) in enumerate(self.spec)}

    def allocate(self, scores: dict) -> dict:
        """The W2 -> W3 allocation on the post-BiIP sensitivity s' = tr(H_G') tr(H_X')."""
        return allocate_bits({n: scores[n][5] for n in scores}, self.params, self.low, self.high, self.budget)

    def quantize(self, W: dict, sign_u: dict, sign_v: dict, bits: dict, stream) -> None:
        """Each sublayer's rotations, Cholesky and sweep at its allocated width; sublayer i
        runs on lane i mod lanes (lanes run concurrently, each in order)."""
        start = torch.cuda.Event()
        start.record(stream)
        for ls in self.lane_streams:
            ls.wait_event(start)
        for i, (name, grp, _, _) in enumerate(self.spec):
            p = self.pipes[name]
            p.bits = bits[name]
            p.run_from_factors(self.HX[grp], self.HG[name], W[name], sign_u[name], sign_v[name],
                               stream=self.lane_streams[i % self.lanes], scales_ready=True)
        for ls in self.lane_streams:
            stream.wait_stream(ls)

    def run(self, X: dict, G: dict, W: dict, sign_u: dict, sign_v: dict, stream=None) -> tuple[dict, dict]:
        """The whole block; returns (bits, scores). Codes, scales and zeros are in
        self.pipes[name].codes / .scale / .zero."""
        s = torch.cuda.current_stream() if stream is None else stream
        self.factors(X, G, s)
        sc = self.scores(W, s)
        bits = self.allocate(sc)
        self.quantize(W, sign_u, sign_v, bits, s)
        return bits, sc

    def check(self) -> None:
        """Raise the first device-side error of the block; every word is read and cleared."""
        torch.cuda.synchronize()
        st, raw = kq.kq_check(self.info, reset=True)
        first = None if st == kq.KQ_OK else kq.KronqError(st, "block", f"device word {raw}")
        for p in self.pipes.values():
            try:
                p.check()
            except kq.KronqError as e:
                first = first or e
        if first is not None:
            raise first
