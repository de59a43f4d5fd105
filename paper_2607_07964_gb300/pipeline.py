"""One linear layer through the four stages of the KronQ path (Algorithms 1 and 2), as a
sequence of libkronq calls on one or two CUDA streams: GPTQ mode, or with the GPTAQ drift
correction (the full objective of Eq. kronq_full) when a scaling alpha is given and the
full-precision input X~ is passed to run(). Buffers and workspaces are allocated once
(torch provides the device memory) and reused across layers of the same shape.
"""
from __future__ import annotations

import torch

from . import kronq as kq

STAGES = ("factor_x", "factor_g", "scales_traces", "rotate", "chol", "sweep")
# with the drift correction: the drift statistic after H_X, and P after the Cholesky
STAGES_DRIFT = ("factor_x", "drift", "factor_g", "scales_traces", "rotate", "chol", "p", "sweep")


class PriorityGraph:
    """A captured torch graph (keep_graph=True) instantiated by the library with its
    per-node priorities; replay() launches it on the current stream."""

    def __init__(self, g):
        self.g = g   # keeps the captured graph and its memory pool alive
        self.exec = kq.kq_graph_instantiate(g.raw_cuda_graph(), True)

    def replay(self) -> None:
        kq.kq_graph_launch(self.exec, torch.cuda.current_stream())

    def __del__(self):
        if getattr(self, "exec", None):
            kq.kq_graph_exec_destroy(self.exec)
            self.exec = None


class LayerPipeline:
    """Device buffers for one layer shape and the stage sequence that fills them."""

    def __init__(self, d_out: int, d_in: int, bits: int, group: int, block: int = 128,
                 damp: float = 0.01, device: str = "cuda", want_col_loss: bool = True,
                 overlap: bool = True, x_chunk_tokens: int = 0, g_chunk_tokens: int = 32768,
                 trailing: str = "3xtf32", alpha: float | None = None, drift_chunk_tokens: int = 0,
                 debug_outputs: bool = False):
        self.d_out, self.d_in, self.bits, self.group, self.block, self.damp = d_out, d_in, bits, group, block, damp
        # GPTAQ drift correction (Prop. 1, Alg. 2) with scaling alpha; None = GPTQ mode
        self.alpha = alpha
        self.stages = STAGES if alpha is None else STAGES_DRIFT
        f32 = dict(dtype=torch.float32, device=device)
        ng = 1 if group == 0 else -(-d_in // group)
        self.HX = torch.empty((d_in, d_in), **f32)
        self.HG = torch.empty((d_out, d_out), **f32)
        self.Wp = torch.empty((d_out, d_in), **f32)
        self.s_x = torch.empty((d_in,), **f32)
        self.s_g = torch.empty((d_out,), **f32)
        self.Lt = torch.empty((d_in, d_in), **f32)
        self.codes = torch.empty((d_out, d_in), dtype=torch.uint8, device=device)
        self.scale = torch.empty((d_out, ng), **f32)
        self.zero = torch.empty((d_out, ng), dtype=torch.int32, device=device)
        self.col_loss = torch.empty((d_in,), **f32) if want_col_loss else None
        self.traces = torch.zeros((6,), dtype=torch.float64, device=device)
        self.trace_x = torch.zeros((1,), dtype=torch.float64, device=device)
        self.trace_g = torch.zeros((1,), dtype=torch.float64, device=device)
        self.info = torch.zeros((4,), dtype=torch.int32, device=device)
        self.ws_chol = torch.empty((kq.kq_chol_inv_workspace(d_in),), dtype=torch.uint8, device=device)
        # the sweep's lazy trailing update: "fp32" (the fp32-ordered definition, bit-exact) or
        # "3xtf32" (tensor cores, 3xTF32 split)
        self.trail_mode = {"fp32": kq.KQ_TRAIL_FP32, "3xtf32": kq.KQ_TRAIL_3XTF32}[trailing]
        self.ws_obs = torch.empty((kq.kq_obs_quantize_workspace(d_out, d_in, block, self.trail_mode,
                                                                alpha is not None),),
                                  dtype=torch.uint8, device=device)
        # debug outputs (checks only): the rotated W' as the sweep receives it, and the
        # sweep's pre-quantization value of every weight (kq_obs_quantize's pre_q)
        self.Wp_in = torch.empty((d_out, d_in), **f32) if debug_outputs else None
        self.pre_q = torch.empty((d_out, d_in), **f32) if debug_outputs else None
        if alpha is not None:
            self.D = torch.empty((d_in, d_in), **f32)      # drift statistic, then D'
            self.Pt = torch.empty((d_in, d_in), **f32)
            self.ws_p = torch.empty((kq.kq_gptaq_p_workspace(d_in),), dtype=torch.uint8, device=device)
        else:
            self.D = self.Pt = None
        # the split drift of this many tokens at a time (0: all tokens of the first run; the
        # call chunks the tokens itself when its workspace holds fewer)
        self.drift_chunk_tokens = drift_chunk_tokens
        self.ws_drift = None
        # Output-side work (H_G, S_G, U) runs on a second stream beside the Cholesky, which
        # needs only H_X and leaves most SMs idle during its diagonal steps.
        # The critical path (H_X, Cholesky, sweep) runs on a high-priority stream so SMs freed
        # by the long-running H_G tiles go to it first.
        self.overlap = overlap
        # H_X and H_G are accumulated over token chunks of these sizes (0: one call). The host
        # path copies X, then G, and accumulates each chunk as soon as it has arrived; G is
        # the last input, so chunking it hides its accumulation under its own copy, while
        # H_X's single call already hides under G's copy. In the device-resident schedule
        # H_G runs on the side stream, where the cost of the shorter calls is mostly hidden.
        self.chunk_tokens = {"X": x_chunk_tokens, "G": g_chunk_tokens}
        try:
            lo, hi = torch.cuda.Stream.priority_range()
        except (AttributeError, RuntimeError):
            lo, hi = 0, -1
        self.main = torch.cuda.Stream(device=device, priority=hi) if overlap else None
        self.side = torch.cuda.Stream(device=device, priority=lo) if overlap else None
        self.copy = None
        self._ev = [torch.cuda.Event() for _ in range(8)]
        # when the low-priority stream may start: at once ("start"), after H_X ("factor") or
        # after the input-side rotation ("rotate"); measured on q_proj, runs alternated:
        # GPTQ mode 6.28 ms ("rotate") against 6.47 ("start"), with the drift correction
        # 13.76 ms ("factor") against 13.89 ("rotate")
        self.side_after = "rotate" if alpha is None else "factor"

    def _chunks(self, which: str, T: int) -> list[tuple[int, int]]:
        c = self.chunk_tokens[which]
        c = c if c > 0 else max(T, 1)
        ch = [(t0, min(T, t0 + c)) for t0 in range(0, max(T, 1), c)]
        if which == "X" and self.chunk_tokens["X"] > 0 and len(ch) > 1:
            # the first chunk in four: on the host path the accumulation of H_X starts once a
            # quarter chunk has arrived (the later chunks arrive faster than they are summed)
            t0, t1 = ch.pop(0)
            q = max(1, -(-(t1 - t0) // 4))
            ch = [(a, min(t1, a + q)) for a in range(t0, t1, q)] + ch
        if which == "G" and self.chunk_tokens["G"] > 0 and len(ch) > 1:
            # the last chunk in four: after G's last bytes arrive on the host path, only a
            # quarter chunk of accumulation stands before S_G, U and the sweep
            t0, t1 = ch.pop()
            q = max(1, -(-(t1 - t0) // 4))
            ch += [(a, min(t1, a + q)) for a in range(t0, t1, q)]
        return ch

    def _factor(self, which, A, H, trace, info, stream, ready=None) -> None:
        """H = A^T A over the token chunks (Alg. 1 online statistic); `ready`, if given,
        holds one event per chunk that the stream waits on before using it."""
        ch = self._chunks(which, A.shape[0])
        for c, (t0, t1) in enumerate(ch):
            if ready is not None:
                stream.wait_event(ready[c])
            kq.kq_accum_factor(A[t0:t1], H, accumulate=c > 0, trace=trace if c == len(ch) - 1 else None,
                               info=info, stream=stream)

    def _need_xt(self, Xt) -> None:
        if (self.alpha is None) != (Xt is None):
            raise ValueError("X~ must be given exactly when the pipeline has a drift scaling alpha")
        if Xt is not None and self.ws_drift is None:   # sized once, before any graph capture
            tokens = self.drift_chunk_tokens if self.drift_chunk_tokens > 0 else Xt.shape[0]
            self.ws_drift = torch.empty((kq.kq_accum_drift_workspace(tokens, self.d_in),), dtype=torch.uint8,
                                        device=self.HX.device)

    def run(self, X, G, W, sign_u, sign_v, stream=None, events=None, Xt=None) -> None:
        """X [T, d_in] bf16, G [T, d_out] bf16, W [d_out, d_in] fp32 (left unchanged), signs
        int8; Xt = X~ [T, d_in] bf16 with the drift correction. `events`, if given, is a list
        of len(self.stages) + 1 CUDA events recorded at the stage boundaries on the stream."""
        self._need_xt(Xt)
        s = torch.cuda.current_stream() if stream is None else stream
        if self.overlap and events is None:
            self._run_overlapped(X, G, W, sign_u, sign_v, s, Xt=Xt)
            return
        marks = iter(range(len(self.stages) + 1))

        def mark():
            # stage boundary: an event (if asked) and an NVTX range named after the stage
            i = next(marks)
            if events is not None:
                events[i].record(s)
            if i > 0:
                torch.cuda.nvtx.range_pop()
            if i < len(self.stages):
                torch.cuda.nvtx.range_push(f"kronq.{self.stages[i]}")

        mark()
        self._factor("X", X, self.HX, self.trace_x, self.info[0:1], s)                           # Alg. 1: H_X
        mark()
        if Xt is not None:                                                                        # Alg. 1: Delta X X^T
            kq.kq_accum_drift(Xt, X, self.D, info=self.info[0:1], ws=self.ws_drift, stream=s)
            mark()
        self._factor("G", G, self.HG, self.trace_g, self.info[2:3], s)                           # H_G
        mark()
        kq.kq_compute_scales(W, self.HX, self.HG, self.s_x, self.s_g, stream=s)          # Eq. (rescale)
        kq.kq_traces(self.HX, self.s_x, self.HG, self.s_g, self.traces, stream=s)         # Eq. (sensitivity)
        mark()
        with torch.cuda.stream(s):
            self.Wp.copy_(W)
        kq.kq_rotate_in(self.Wp, self.HX, self.s_x, sign_v, kq.KQ_FWD_SYM, stream=s)         # Eq. (biip), V side
        if Xt is not None:
            kq.kq_rotate_in(None, self.D, self.s_x, sign_v, kq.KQ_FWD, stream=s)         # D' = V S^-1 D S^-1 V^T
        kq.kq_rotate_out(self.Wp, None, self.s_g, sign_u, kq.KQ_FWD, stream=s)           # U side
        kq.kq_rotate_out(None, self.HG, self.s_g, sign_u, kq.KQ_FWD_SYM, stream=s)           # H_G, then released
        mark()
        kq.kq_chol_inv(self.HX, self.damp, self.Lt, self.info[1:2], self.ws_chol, stream=s)  # Alg. 2
        mark()
        if Xt is not None:
            kq.kq_gptaq_p(self.D, self.Lt, self.alpha, self.Pt, self.ws_p, info=self.info[1:2], stream=s)  # P
            mark()
        self._sweep(s, Xt is not None)                                                   # Alg. 2 sweep
        mark()

    def _sweep(self, stream, with_p: bool) -> None:
        """Algorithm 2's sweep on W' (destroyed) with L; the debug copies first if asked."""
        if self.Wp_in is not None:
            with torch.cuda.stream(stream):
                self.Wp_in.copy_(self.Wp)
        kq.kq_obs_quantize(self.Wp, self.Lt, self.bits, self.group, self.block, self.codes, self.scale,
                           self.zero, self.col_loss, self.pre_q, self.ws_obs, stream=stream, mode=self.trail_mode,
                           info=self.info[3:4], Pt=self.Pt if with_p else None)

    def _run_overlapped(self, X, G, W, sign_u, sign_v, caller, x_ready=None, g_ready=None, w_ready=None,
                        Xt=None, xt_ready=None) -> None:
        """The same results on two streams. The Cholesky needs only H_X and leaves most SMs
        idle during its diagonal steps, so H_G, S_G and U go to a low-priority stream that
        runs beside it; the high-priority stream does H_X, S_X, V, the Cholesky and (once
        U is applied to W) the sweep, while H_G's own rotation finishes beside the sweep.
        With the drift correction the drift statistic and its rotation run first on the
        low-priority stream, and P on the high-priority one after the Cholesky.
        Events order the shared buffers; x_ready / g_ready / w_ready / xt_ready are the host
        path's copy events."""
        torch.cuda.nvtx.range_push("kronq.layer")
        try:
            self._enqueue_overlapped(X, G, W, sign_u, sign_v, caller, x_ready, g_ready, w_ready, Xt, xt_ready)
        finally:
            torch.cuda.nvtx.range_pop()

    def _enqueue_overlapped(self, X, G, W, sign_u, sign_v, caller, x_ready, g_ready, w_ready, Xt, xt_ready) -> None:
        s, s2 = self.main, self.side
        e_in, e_fx, e_tx, e_rin, e_side, e_out, e_hg, e_d = self._ev
        e_in.record(caller)
        s.wait_event(e_in)
        s2.wait_event(e_in)
        self._factor("X", X, self.HX, self.trace_x, self.info[0:1], s, x_ready)
        e_fx.record(s)
        if w_ready is not None:
            s.wait_event(w_ready)
        kq.kq_compute_scales(W, self.HX, None, self.s_x, None, stream=s)
        kq.kq_traces(self.HX, self.s_x, None, None, self.traces, stream=s)
        e_tx.record(s)
        with torch.cuda.stream(s):
            self.Wp.copy_(W)
        kq.kq_rotate_in(self.Wp, self.HX, self.s_x, sign_v, kq.KQ_FWD_SYM, stream=s)
        e_rin.record(s)
        kq.kq_chol_inv(self.HX, self.damp, self.Lt, self.info[1:2], self.ws_chol, stream=s)
        # When the low-priority stream starts (side_after): its long tensor-core tiles hold
        # SMs the rotation and the Cholesky then wait for.
        if self.side_after != "start":
            s2.wait_event(e_rin if self.side_after == "rotate" else e_fx)
        if Xt is not None:
            if xt_ready is not None:
                s2.wait_event(xt_ready)
            kq.kq_accum_drift(Xt, X, self.D, info=self.info[2:3], ws=self.ws_drift, stream=s2)
            kq.kq_rotate_in(None, self.D, self.s_x, sign_v, kq.KQ_FWD, stream=s2)
            e_d.record(s2)
        self._factor("G", G, self.HG, self.trace_g, self.info[2:3], s2, g_ready)
        s2.wait_event(e_tx)                      # W (host path) and the X side of the traces
        kq.kq_compute_scales(W, None, self.HG, None, self.s_g, stream=s2)
        kq.kq_traces(None, None, self.HG, self.s_g, self.traces, stream=s2)
        s2.wait_event(e_rin)
        kq.kq_rotate_out(self.Wp, None, self.s_g, sign_u, kq.KQ_FWD, stream=s2)
        e_side.record(s2)
        kq.kq_rotate_out(None, self.HG, self.s_g, sign_u, kq.KQ_FWD_SYM, stream=s2)
        e_hg.record(s2)
        if Xt is not None:
            s.wait_event(e_d)
            kq.kq_gptaq_p(self.D, self.Lt, self.alpha, self.Pt, self.ws_p, info=self.info[1:2], stream=s)
        s.wait_event(e_side)
        self._sweep(s, Xt is not None)
        e_out.record(s)
        caller.wait_event(e_out)
        caller.wait_event(e_hg)

    def run_from_factors(self, HX_raw, HG_raw, W, sign_u, sign_v, stream=None, scales_ready: bool = False) -> None:
        """Stages 2-4 from factors accumulated elsewhere (a factor shared by several
        sublayers, Sec. 3.3: q, k and v read the same input). HX_raw / HG_raw are copied
        into this pipeline's buffers (the rotations work in place). scales_ready: s_x, s_g
        and the traces are already in this pipeline's buffers (computed from the same raw
        factors). The Cholesky runs on this pipeline's high-priority stream with the H_G
        side beside it, as in run()."""
        s = torch.cuda.current_stream() if stream is None else stream
        main = self.main if self.overlap else s
        side = self.side if self.overlap else s
        e_in, e_fx, e_tx, e_rin, e_side, e_out, e_hg, _ = self._ev
        e_in.record(s)
        main.wait_event(e_in)
        side.wait_event(e_in)
        with torch.cuda.stream(main):
            self.HX.copy_(HX_raw)
        if not scales_ready:
            kq.kq_compute_scales(W, self.HX, None, self.s_x, None, stream=main)
            kq.kq_traces(self.HX, self.s_x, None, None, self.traces, stream=main)
        e_tx.record(main)
        with torch.cuda.stream(main):
            self.Wp.copy_(W)
        kq.kq_rotate_in(self.Wp, self.HX, self.s_x, sign_v, kq.KQ_FWD_SYM, stream=main)
        e_rin.record(main)
        kq.kq_chol_inv(self.HX, self.damp, self.Lt, self.info[1:2], self.ws_chol, stream=main)
        with torch.cuda.stream(side):
            self.HG.copy_(HG_raw)
        side.wait_event(e_tx)
        if not scales_ready:
            kq.kq_compute_scales(W, None, self.HG, None, self.s_g, stream=side)
            kq.kq_traces(None, None, self.HG, self.s_g, self.traces, stream=side)
        side.wait_event(e_rin)
        kq.kq_rotate_out(self.Wp, None, self.s_g, sign_u, kq.KQ_FWD, stream=side)
        e_side.record(side)
        kq.kq_rotate_out(None, self.HG, self.s_g, sign_u, kq.KQ_FWD_SYM, stream=side)
        e_hg.record(side)
        main.wait_event(e_side)
        self._sweep(main, False)
        e_out.record(main)
        s.wait_event(e_out)
        s.wait_event(e_hg)

    def capture(self, X, G, W, sign_u, sign_v, Xt=None) -> tuple:
        """Record one layer (both streams) as a CUDA graph on these fixed buffers. Returns
        (graph, kernels per replay); graph.replay() launches it on the current stream. Run
        run() once first so one-time set-up is done. The graph is instantiated with the
        priorities its kernels were captured with (critical path above side work), where
        this PyTorch exposes the captured graph."""
        from . import kronq as _kq
        torch.cuda.synchronize()
        try:
            g = torch.cuda.CUDAGraph(keep_graph=True)
        except TypeError:
            g = None
        plain = g is None
        if plain:
            g = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream(device=self.HX.device)
        n0 = _kq.launch_count()
        with torch.cuda.graph(g, stream=cap):
            self.run(X, G, W, sign_u, sign_v, stream=cap, Xt=Xt)
        n = _kq.launch_count() - n0
        return (g if plain else PriorityGraph(g)), n

    def check(self, stream=None) -> None:
        """Raise if a kernel reported a device-side error (timeout, non-PD pivot)."""
        if self.side is not None:
            self.side.synchronize()
            self.main.synchronize()
        # read (and clear) every word first, so that no stale report survives the raise
        found = [kq.kq_check(self.info[k:k + 1], reset=True, stream=stream) for k in range(4)]
        for st, raw in found:
            if st != kq.KQ_OK:
                raise kq.KronqError(st, "pipeline", f"device word {raw}")

    def run_host(self, X_h, G_h, W_h, su_h, sv_h, codes_h, scale_h, zero_h, stream=None, Xt_h=None) -> tuple[int, int]:
        """End-to-end call with HOST buffers (pinned for asynchronous copies): copy the
        layer's inputs to the device, run the four stages, copy codes and grids back.
        Enqueued on `stream`; the caller synchronizes. Returns (bytes in, bytes out).

        The copies run on their own stream in the order X chunks, W, signs, G chunks (W is
        first needed after H_X), and each chunk's factor accumulation starts as soon as that
        chunk has arrived, so the host link overlaps the factor, rescale, rotation and
        Cholesky work; without the two-stream schedule the copies simply precede the run."""
        self._need_xt(Xt_h)
        s = torch.cuda.current_stream() if stream is None else stream
        dev = self.HX.device
        if getattr(self, "_stage", None) is None or self._stage["X"].shape != X_h.shape or \
                (Xt_h is not None) != ("Xt" in self._stage):
            self._stage = {
                "X": torch.empty(X_h.shape, dtype=X_h.dtype, device=dev),
                "G": torch.empty(G_h.shape, dtype=G_h.dtype, device=dev),
                "W": torch.empty(W_h.shape, dtype=W_h.dtype, device=dev),
                "su": torch.empty(su_h.shape, dtype=su_h.dtype, device=dev),
                "sv": torch.empty(sv_h.shape, dtype=sv_h.dtype, device=dev),
            }
            if Xt_h is not None:
                self._stage["Xt"] = torch.empty(Xt_h.shape, dtype=Xt_h.dtype, device=dev)
        st = self._stage
        ins = [X_h, G_h, W_h, su_h, sv_h] + ([] if Xt_h is None else [Xt_h])
        nin = sum(t.numel() * t.element_size() for t in ins)
        nout = sum(t.numel() * t.element_size() for t in (codes_h, scale_h, zero_h))
        if not self.overlap:
            with torch.cuda.stream(s):
                pairs = [("X", X_h), ("G", G_h), ("W", W_h), ("su", su_h), ("sv", sv_h)]
                for k, h in pairs + ([] if Xt_h is None else [("Xt", Xt_h)]):
                    st[k].copy_(h, non_blocking=True)
            self.run(st["X"], st["G"], st["W"], st["su"], st["sv"], stream=s, Xt=st.get("Xt"))
        else:
            if self.copy is None:
                self.copy = torch.cuda.Stream(device=dev)
            cs = self.copy
            e0 = torch.cuda.Event()
            e0.record(s)
            cs.wait_event(e0)
            with torch.cuda.stream(cs):
                ready = {}
                for k, h in (("X", X_h), ("G", G_h)):
                    ready[k] = []
                    for t0, t1 in self._chunks(k, h.shape[0]):
                        st[k][t0:t1].copy_(h[t0:t1], non_blocking=True)
                        ev = torch.cuda.Event()
                        ev.record(cs)
                        ready[k].append(ev)
                    if k == "X":
                        if Xt_h is not None:   # X~ right after X: the drift needs both
                            st["Xt"].copy_(Xt_h, non_blocking=True)
                            xt_ready = torch.cuda.Event()
                            xt_ready.record(cs)
                        for kk, hh in (("W", W_h), ("su", su_h), ("sv", sv_h)):
                            st[kk].copy_(hh, non_blocking=True)
                        w_ready = torch.cuda.Event()
                        w_ready.record(cs)
            self._run_overlapped(st["X"], st["G"], st["W"], st["su"], st["sv"], s, x_ready=ready["X"],
                                 g_ready=ready["G"], w_ready=w_ready, Xt=st.get("Xt"),
                                 xt_ready=xt_ready if Xt_h is not None else None)
        with torch.cuda.stream(s):
            codes_h.copy_(self.codes, non_blocking=True)
            scale_h.copy_(self.scale, non_blocking=True)
            zero_h.copy_(self.zero, non_blocking=True)
        return nin, nout
