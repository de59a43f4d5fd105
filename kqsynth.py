"""Seeded synthetic inputs for one linear layer (weights, calibration activations,
output gradients, RHT sign vectors).

This module is shared by the tests, the oracle's callers and the benchmark. It holds
none of the quantization method's arithmetic: it only draws random numbers with a fixed
recipe and rounds them to the storage types the method consumes.

Recipe (stands in for the paper's 128 x 2048-token WikiText-2 calibration set and for
Llama weights, Sec. 5.1; neither is available here):
  * activations x[t, j] = sigma_j * z, sigma_j = exp(N(0, 1)); the first `n_outliers`
    entries of a seeded permutation of the channels are multiplied by 20;
  * gradients   g[t, i] = tau_i * z, tau_i = exp(N(0, g_sigma^2));
  * weights     W[i, j] = 0.02 * z, each entry multiplied by 10 with probability 0.001;
  * X and G are rounded to bf16 (round-to-nearest-even); W is rounded to bf16 unless
    `w_bf16` is False (then it stays fp32);
  * RHT sign vectors are +-1 (int8), one per side;
  * for the GPTAQ drift correction, the full-precision model's input is
    x~[t, j] = x[t, j] + drift * sigma_j * z (drift = 0.1 by default), rounded to bf16: X is
    read as the running quantized model's input and X~ - X as its drift.
Every tensor has its own sub-seed, so changing one shape does not change the others.
"""
from __future__ import annotations

import dataclasses

import numpy as np

_SUB = {"xscale": 1, "xperm": 2, "x": 3, "gscale": 4, "g": 5, "w": 6, "wbern": 7,
        "sign_u": 8, "sign_v": 9, "xdrift": 10}


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    """Shape and quantizer settings of one synthetic linear layer."""
    name: str
    d_out: int
    d_in: int
    T: int
    bits: int
    group: int          # 0 = one grid per output row, else the group width (== block)
    n_outliers: int
    g_sigma: float
    w_bf16: bool = True
    block: int = 128
    damp: float = 0.01
    seed: int = 0

    def replace(self, **kw) -> "LayerConfig":
        return dataclasses.replace(self, **kw)


# Llama-shaped layers. The first is the small case the oracle finishes in seconds; the
# second is the 8B q_proj the benchmark times by default.
CONFIGS = {
    "tiny256": LayerConfig("tiny256", 256, 256, 4096, 4, 0, 4, 1.0, w_bf16=False),
    "q_proj_8b": LayerConfig("q_proj_8b", 4096, 4096, 131072, 4, 128, 16, 1.5),
    "gate_up_8b": LayerConfig("gate_up_8b", 14336, 4096, 262144, 3, 128, 16, 1.5),
    "down_8b": LayerConfig("down_8b", 4096, 14336, 262144, 3, 128, 16, 1.5),
    "qo_70b": LayerConfig("qo_70b", 8192, 8192, 262144, 2, 128, 16, 1.5),
    "kv_70b": LayerConfig("kv_70b", 1024, 8192, 262144, 2, 128, 16, 1.5),
    "down_70b": LayerConfig("down_70b", 8192, 28672, 262144, 2, 128, 64, 1.5),
}


def _rng(seed: int, what: str) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(key=[seed, _SUB[what]]))


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round finite float32 values to the nearest bf16 (ties to even); returns float32."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).copy()
    u += np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    u &= np.uint32(0xFFFF0000)
    return u.view(np.float32)


def _scaled_normals(rng: np.random.Generator, T: int, d: int, scale: np.ndarray) -> np.ndarray:
    """bf16-rounded N(0,1) * scale, drawn in row chunks (same stream as one draw)."""
    out = np.empty((T, d), dtype=np.float32)
    step = max(1, (1 << 24) // max(d, 1))
    for t0 in range(0, T, step):
        t1 = min(T, t0 + step)
        z = rng.standard_normal((t1 - t0, d), dtype=np.float32)
        z *= scale[None, :]
        out[t0:t1] = round_bf16(z)
    return out


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """Upper 16 bits of float32 values that are exactly representable in bf16."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    return (a.view(np.uint32) >> 16).astype(np.uint16)


def channel_scales(cfg: LayerConfig) -> tuple[np.ndarray, np.ndarray]:
    """Per-channel std of the activations (d_in) and of the gradients (d_out)."""
    sx = np.exp(_rng(cfg.seed, "xscale").standard_normal(cfg.d_in))
    perm = _rng(cfg.seed, "xperm").permutation(cfg.d_in)
    sx[perm[: cfg.n_outliers]] *= 20.0
    sg = np.exp(cfg.g_sigma * _rng(cfg.seed, "gscale").standard_normal(cfg.d_out))
    return sx.astype(np.float32), sg.astype(np.float32)


def activations(cfg: LayerConfig, T: int | None = None) -> np.ndarray:
    """X [T, d_in], bf16-representable float32, tokens as rows."""
    T = cfg.T if T is None else T
    sx, _ = channel_scales(cfg)
    return _scaled_normals(_rng(cfg.seed, "x"), T, cfg.d_in, sx)


def fp_activations(cfg: LayerConfig, X: np.ndarray, drift: float = 0.1) -> np.ndarray:
    """X~ [T, d_in] = bf16(X + drift * sigma_j * z): the full-precision model's input to the
    layer whose running quantized input is X (bf16-representable float32)."""
    sx, _ = channel_scales(cfg)
    T = X.shape[0]
    noise = _scaled_normals(_rng(cfg.seed, "xdrift"), T, cfg.d_in, (drift * sx).astype(np.float32))
    return round_bf16(np.asarray(X, np.float32) + noise)


def gradients(cfg: LayerConfig, T: int | None = None) -> np.ndarray:
    """G [T, d_out], bf16-representable float32, tokens as rows."""
    T = cfg.T if T is None else T
    _, sg = channel_scales(cfg)
    return _scaled_normals(_rng(cfg.seed, "g"), T, cfg.d_out, sg)


def weights(cfg: LayerConfig) -> np.ndarray:
    """W [d_out, d_in] float32 (bf16-representable when cfg.w_bf16)."""
    w = 0.02 * _rng(cfg.seed, "w").standard_normal((cfg.d_out, cfg.d_in), dtype=np.float32)
    big = _rng(cfg.seed, "wbern").random((cfg.d_out, cfg.d_in)) < 0.001
    w = np.where(big, w * 10.0, w).astype(np.float32)
    return round_bf16(w) if cfg.w_bf16 else w


def signs(cfg: LayerConfig) -> tuple[np.ndarray, np.ndarray]:
    """RHT sign vectors (sigma_U of length d_out, sigma_V of length d_in), int8 +-1."""
    su = np.where(_rng(cfg.seed, "sign_u").random(cfg.d_out) < 0.5, -1, 1).astype(np.int8)
    sv = np.where(_rng(cfg.seed, "sign_v").random(cfg.d_in) < 0.5, -1, 1).astype(np.int8)
    return su, sv


def layer(cfg: LayerConfig, T: int | None = None) -> dict:
    """All host inputs of one layer."""
    su, sv = signs(cfg)
    return {"X": activations(cfg, T), "G": gradients(cfg, T), "W": weights(cfg),
            "sign_u": su, "sign_v": sv}


def random_spd(n: int, seed: int, cond_decay: float = 3.0) -> np.ndarray:
    """A seeded symmetric positive-definite float64 matrix shaped like a calibration
    second-moment matrix: B^T B over 4n random tokens with lognormal channel scales."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 101]))
    sc = np.exp(rng.standard_normal(n) * cond_decay / 3.0)
    b = rng.standard_normal((4 * n, n)) * sc[None, :]
    return b.T @ b


def device_layer(cfg: LayerConfig, device: str = "cuda"):
    """The same recipe drawn on the GPU with torch's generator (used where the host
    generator would take minutes). Values differ from `layer`, distribution is equal."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(cfg.seed * 7919 + 17)
    sx, sg = channel_scales(cfg)
    sx_t = torch.from_numpy(sx).to(device)
    sg_t = torch.from_numpy(sg).to(device)
    X = torch.empty((cfg.T, cfg.d_in), dtype=torch.bfloat16, device=device)
    G = torch.empty((cfg.T, cfg.d_out), dtype=torch.bfloat16, device=device)
    chunk = max(1, (1 << 26) // max(cfg.d_in, cfg.d_out))
    for t0 in range(0, cfg.T, chunk):
        t1 = min(cfg.T, t0 + chunk)
        z = torch.randn((t1 - t0, cfg.d_in), generator=gen, device=device)
        X[t0:t1] = (z * sx_t).to(torch.bfloat16)
        z = torch.randn((t1 - t0, cfg.d_out), generator=gen, device=device)
        G[t0:t1] = (z * sg_t).to(torch.bfloat16)
    w = 0.02 * torch.randn((cfg.d_out, cfg.d_in), generator=gen, device=device)
    big = torch.rand((cfg.d_out, cfg.d_in), generator=gen, device=device) < 0.001
    w = torch.where(big, w * 10.0, w)
    if cfg.w_bf16:
        w = w.to(torch.bfloat16).float()
    su, sv = signs(cfg)
    return {"X": X, "G": G, "W": w.contiguous(),
            "sign_u": torch.from_numpy(su).to(device), "sign_v": torch.from_numpy(sv).to(device)}


def device_fp_activations(cfg: LayerConfig, X, drift: float = 0.1):
    """X~ = bf16(X + drift * sigma_j * z) drawn on the GPU with torch's generator (the device
    counterpart of `fp_activations`)."""
    import torch

    gen = torch.Generator(device=X.device)
    gen.manual_seed(cfg.seed * 7919 + 23)
    sx, _ = channel_scales(cfg)
    sx_t = torch.from_numpy(drift * sx).to(X.device)
    Xt = torch.empty_like(X)
    chunk = max(1, (1 << 26) // cfg.d_in)
    for t0 in range(0, X.shape[0], chunk):
        t1 = min(X.shape[0], t0 + chunk)
        z = torch.randn((t1 - t0, cfg.d_in), generator=gen, device=X.device)
        Xt[t0:t1] = (X[t0:t1].float() + z * sx_t).to(torch.bfloat16)
    return Xt


# ------------------------------------------------------------------ transformer blocks
@dataclasses.dataclass(frozen=True)
class BlockConfig:
    """One Llama-style transformer block: attention q, k, v (shared input), o, and MLP
    gate, up (shared input), down; the bit widths and the mean-bits budget of the W2 -> W3
    allocation."""
    name: str
    d_model: int
    d_kv: int
    d_ff: int
    T: int
    group: int = 128
    block: int = 128
    damp: float = 0.01
    low_bits: int = 2
    high_bits: int = 3
    budget: float = 2.5
    n_outliers: int = 16
    g_sigma: float = 1.5
    w_bf16: bool = True
    seed: int = 0

    def replace(self, **kw) -> "BlockConfig":
        return dataclasses.replace(self, **kw)


BLOCKS = {
    "tiny_block": BlockConfig("tiny_block", 256, 64, 512, 2048, n_outliers=4),
    "llama3_8b_block": BlockConfig("llama3_8b_block", 4096, 1024, 14336, 131072),
}

INPUTS = ("attn", "o", "mlp", "down")


def block_spec(cfg: BlockConfig) -> list[tuple[str, str, int, int]]:
    """(sublayer, input group, d_out, d_in) of the seven linear sublayers: q, k, v read the
    attention input, gate and up the MLP input."""
    m, kv, ff = cfg.d_model, cfg.d_kv, cfg.d_ff
    return [("q", "attn", m, m), ("k", "attn", kv, m), ("v", "attn", kv, m), ("o", "o", m, m),
            ("gate", "mlp", ff, m), ("up", "mlp", ff, m), ("down", "down", m, ff)]


def _input_dim(cfg: BlockConfig, group: str) -> int:
    return cfg.d_ff if group == "down" else cfg.d_model


def _sub_cfg(cfg: BlockConfig, d_out: int, d_in: int, k: int) -> LayerConfig:
    return LayerConfig(f"{cfg.name}.{k}", d_out, d_in, cfg.T, cfg.low_bits, cfg.group, cfg.n_outliers,
                       cfg.g_sigma, w_bf16=cfg.w_bf16, block=cfg.block, damp=cfg.damp, seed=cfg.seed * 64 + k)


def block_inputs(cfg: BlockConfig) -> dict:
    """Host inputs of a block: X per input group, and G, W, signs per sublayer (each tensor
    drawn from its own sub-seed with the single-layer recipe)."""
    X = {g: activations(_sub_cfg(cfg, 8, _input_dim(cfg, g), 1 + i)) for i, g in enumerate(INPUTS)}
    out = {"X": X, "G": {}, "W": {}, "sign_u": {}, "sign_v": {}}
    for k, (name, _, d_out, d_in) in enumerate(block_spec(cfg)):
        c = _sub_cfg(cfg, d_out, d_in, 16 + k)
        out["G"][name] = gradients(c)
        out["W"][name] = weights(c)
        out["sign_u"][name], out["sign_v"][name] = signs(c)
    return out


def device_block(cfg: BlockConfig, device: str = "cuda") -> dict:
    """The block's inputs drawn on the GPU (same recipe as block_inputs, torch's generator)."""
    import torch

    X = {}
    for i, g in enumerate(INPUTS):
        X[g] = device_layer(_sub_cfg(cfg, 8, _input_dim(cfg, g), 1 + i), device)["X"]
        torch.cuda.empty_cache()
    out = {"X": X, "G": {}, "W": {}, "sign_u": {}, "sign_v": {}}
    for k, (name, _, d_out, d_in) in enumerate(block_spec(cfg)):
        d = device_layer(_sub_cfg(cfg, d_out, d_in, 16 + k).replace(T=cfg.T), device)
        out["G"][name], out["W"][name] = d["G"], d["W"]
        out["sign_u"][name], out["sign_v"][name] = d["sign_u"], d["sign_v"]
        del d
        torch.cuda.empty_cache()
    return out
