"""One linear layer sharded over the ranks of a process group.

The calibration statistics are sums over tokens (Alg. 1's online statistics, H_X = X^T X
and H_G = G^T G), and the rows of W' are independent once R = L^T is fixed (Alg. 2's
column loop updates each row from its own errors), so one layer splits across N GPUs with
exactly two exchange steps:
  * stage 1: tokens split into N contiguous ranges; each rank accumulates H_X and H_G over
    its range, then one all-reduce (sum) of each fp32 factor;
  * stages 2 and 3 (rescale, rotations, inverse Cholesky): every rank computes them from
    the same reduced factors with the same kernels, so every rank holds the same W', L;
  * stage 4: rows split into N contiguous ranges; each rank sweeps its rows, then one
    all-gather of codes, scales and zero points.
Nothing else crosses ranks: no collective runs inside a kernel and no kernel waits on
another rank. The compute goes through a backend object; the default one is the CUDA
library (libkronq through `kronq`), which has no CPU fallback.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def split_range(n: int, rank: int, world: int) -> tuple[int, int]:
    """Rank's contiguous share [a, b) of n items: ceil(n / world) each, the last ones short."""
    per = -(-n // world)
    a = min(n, rank * per)
    return a, min(n, a + per)


class CudaBackend:
    """The layer's stages as libkronq calls on CUDA tensors (the product path)."""

    def __init__(self, d_out: int, d_in: int, bits: int, group: int, block: int, damp: float, device: str,
                 trailing: str = "3xtf32"):
        from . import kronq as kq
        self.kq = kq
        self.d_out, self.d_in, self.bits, self.group, self.block, self.damp = d_out, d_in, bits, group, block, damp
        self.device = device
        self.mode = {"fp32": kq.KQ_TRAIL_FP32, "3xtf32": kq.KQ_TRAIL_3XTF32}[trailing]
        self.ws_chol = torch.empty((kq.kq_chol_inv_workspace(d_in),), dtype=torch.uint8, device=device)
        self.info = torch.zeros((4,), dtype=torch.int32, device=device)

    def factor(self, A: torch.Tensor) -> torch.Tensor:
        d = A.shape[1]
        H = torch.empty((d, d), dtype=torch.float32, device=self.device)
        self.kq.kq_accum_factor(A, H, info=self.info[0:1])
        return H

    def stages_2_3(self, W, HX, HG, sign_u, sign_v):
        """S_X, S_G (Eq. rescale), W' = U S_G W S_X V^T, H_X' (Eq. biip), L (Alg. 2)."""
        kq = self.kq
        s_x = torch.empty((self.d_in,), dtype=torch.float32, device=self.device)
        s_g = torch.empty((self.d_out,), dtype=torch.float32, device=self.device)
        kq.kq_compute_scales(W, HX, HG, s_x, s_g)
        Wp = W.clone()
        kq.kq_rotate_in(Wp, HX, s_x, sign_v, kq.KQ_FWD_SYM)
        kq.kq_rotate_out(Wp, None, s_g, sign_u, kq.KQ_FWD)
        Lt = torch.empty((self.d_in, self.d_in), dtype=torch.float32, device=self.device)
        kq.kq_chol_inv(HX, self.damp, Lt, self.info[1:2], self.ws_chol)
        return Wp, Lt

    def sweep(self, Wp_rows: torch.Tensor, Lt: torch.Tensor):
        """Codes, scale, zero of the given rows of W' (left unchanged: the sweep works on a
        copy, since kq_obs_quantize consumes its W)."""
        kq = self.kq
        m = Wp_rows.shape[0]
        ng = 1 if self.group == 0 else -(-self.d_in // self.group)
        codes = torch.empty((m, self.d_in), dtype=torch.uint8, device=self.device)
        scale = torch.empty((m, ng), dtype=torch.float32, device=self.device)
        zero = torch.empty((m, ng), dtype=torch.int32, device=self.device)
        if m > 0:
            ws = torch.empty((kq.kq_obs_quantize_workspace(m, self.d_in, self.block, self.mode),), dtype=torch.uint8,
                             device=self.device)
            work = Wp_rows.clone(memory_format=torch.contiguous_format)
            kq.kq_obs_quantize(work, Lt, self.bits, self.group, self.block, codes, scale, zero, None, None, ws,
                               mode=self.mode, info=self.info[3:4])
        return codes, scale, zero

    def check(self) -> None:
        torch.cuda.synchronize()
        for k in range(4):
            st, raw = self.kq.kq_check(self.info[k:k + 1])
            if st != self.kq.KQ_OK:
                raise self.kq.KronqError(st, "sharded layer", f"device word {raw}")


class ShardedLayer:
    """Token-split factors, replicated stages 2-3, row-split sweep (module docstring)."""

    def __init__(self, backend, group=None):
        self.backend = backend
        self.group = group

    def _world(self) -> tuple[int, int]:
        if not dist.is_available() or not dist.is_initialized():
            return 0, 1
        return dist.get_rank(self.group), dist.get_world_size(self.group)

    def factors(self, X_local, G_local):
        """H_X, H_G over all ranks' tokens: local sums, then one all-reduce each."""
        HX = self.backend.factor(X_local)
        HG = self.backend.factor(G_local)
        _, world = self._world()
        if world > 1:
            dist.all_reduce(HX, op=dist.ReduceOp.SUM, group=self.group)
            dist.all_reduce(HG, op=dist.ReduceOp.SUM, group=self.group)
        return HX, HG

    def gather_rows(self, part: torch.Tensor, n_rows: int) -> torch.Tensor:
        """The full [n_rows, ...] tensor from every rank's contiguous row range (padded to the
        common share for the all-gather, then trimmed)."""
        rank, world = self._world()
        if world == 1:
            return part
        per = -(-n_rows // world)
        pad = torch.zeros((per,) + tuple(part.shape[1:]), dtype=part.dtype, device=part.device)
        pad[:part.shape[0]] = part
        bufs = [torch.empty_like(pad) for _ in range(world)]
        dist.all_gather(bufs, pad, group=self.group)
        out = [b[:split_range(n_rows, r, world)[1] - split_range(n_rows, r, world)[0]] for r, b in enumerate(bufs)]
        return torch.cat(out, dim=0)

    def run(self, X_local, G_local, W, sign_u, sign_v):
        """X_local / G_local: this rank's token range of X and G; W [d_out, d_in] and the signs
        the same on every rank. Returns the full codes, scale and zero on every rank."""
        HX, HG = self.factors(X_local, G_local)
        Wp, Lt = self.backend.stages_2_3(W, HX, HG, sign_u, sign_v)
        rank, world = self._world()
        d_out = W.shape[0]
        r0, r1 = split_range(d_out, rank, world)
        codes, scale, zero = self.backend.sweep(Wp[r0:r1], Lt)
        return self.gather_rows(codes, d_out), self.gather_rows(scale, d_out), self.gather_rows(zero, d_out)
