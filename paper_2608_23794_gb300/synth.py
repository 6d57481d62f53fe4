"""Seeded synthetic MoCE layers.

Stand-ins for the activations and learned tables of the paper's workloads
(ResNet-50 bottleneck-entrance projections and a ViT-B feed-forward exit
projection, Sec. 3.1 and Sec. 4.1); no dataset or trained weight is used.
This module draws inputs only. It holds none of the layer's arithmetic, so
both the CUDA path and the CPU oracle may consume what it produces.

Recipe (per layer, one seed):
  * x: N(0,1) draws passed through the preceding activation (ReLU for the
    ResNet shapes, exact-erf GELU for the ViT shape), then rounded to the
    layer's dtype (bf16 by round-to-nearest-even);
  * supports: a random subset of ``support_pool`` channels is drawn once;
    every expert draws k distinct channels from it, uniformly without
    replacement, independently across experts (the random fixed supports of
    Sec. 4.5), so the excluded channels always feed the residual expert;
    rows are left in draw order, not sorted;
  * support logits: N(0,1); gate parameters W1 [k,k], b1 [k], w2 [k], b2:
    N(0, 1/k) (std k^-1/2), biases zero where the workload says so;
  * tau bounds [0.2, 6.0] (Sec. 4.1).
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class LayerConfig:
    name: str
    N: int
    H: int
    W: int
    C_in: int
    C_out: int          # routed experts R; the output has R + 1 channels
    k: int
    dtype: str          # "f32" | "bf16"
    layout: str         # "nhwc" | "nchw"
    activation: str     # "relu" | "gelu"
    support_pool: int   # channels the supports are drawn from
    gate_bias_zero: bool = False
    tau_min: float = 0.2
    tau_max: float = 6.0

    def replace(self, **kw) -> "LayerConfig":
        return dataclasses.replace(self, **kw)

    @property
    def HW(self) -> int:
        return self.H * self.W

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4


def _seven_eighths(c: int) -> int:
    return (7 * c) // 8


# The workloads: a tiny fp32 NCHW case, three ResNet-50 bottleneck-entrance
# ("reduce") projections and the ViT-B token-wise feed-forward exit projection
# as a 1x1 layer over 14x14 tokens, swept over k.
CONFIGS: dict[str, LayerConfig] = {
    "tiny_f32_nchw": LayerConfig("tiny_f32_nchw", 2, 8, 8, 64, 16, 4, "f32", "nchw", "relu", 56,
                                 gate_bias_zero=True),
    "rn50_stage1_reduce": LayerConfig("rn50_stage1_reduce", 64, 56, 56, 256, 64, 16, "bf16",
                                      "nhwc", "relu", _seven_eighths(256)),
    "rn50_stage3_reduce": LayerConfig("rn50_stage3_reduce", 256, 14, 14, 1024, 256, 64, "bf16",
                                      "nhwc", "relu", _seven_eighths(1024)),
    "rn50_stage4_reduce": LayerConfig("rn50_stage4_reduce", 256, 7, 7, 2048, 512, 128, "bf16",
                                      "nhwc", "relu", _seven_eighths(2048)),
}
for _k in (32, 96, 192, 384):
    CONFIGS[f"vitb_ffn_exit_k{_k}"] = LayerConfig(f"vitb_ffn_exit_k{_k}", 64, 14, 14, 3072, 768,
                                                  _k, "bf16", "nhwc", "gelu",
                                                  _seven_eighths(3072))


@dataclass
class SyntheticLayer:
    cfg: LayerConfig
    x: np.ndarray               # float32 values exactly representable in cfg.dtype, cfg.layout
    x_bits: np.ndarray | None   # uint16 bf16 bit patterns (bf16 layers), same shape as x
    support_idx: np.ndarray     # int32 [R, k], rows in draw order
    support_logits: np.ndarray  # float32 [R, k]
    W1: np.ndarray              # float32 [k, k], row j = hidden unit j
    b1: np.ndarray              # float32 [k]
    w2: np.ndarray              # float32 [k]
    b2: np.ndarray              # float32 [1]

    def device_x_host(self) -> np.ndarray:
        """The array whose bytes the device path consumes (uint16 bits or float32)."""
        return self.x_bits if self.x_bits is not None else self.x


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).reshape(-1)
    out = np.empty(u.size, np.uint16)
    step = 1 << 22
    for s0 in range(0, u.size, step):
        v = u[s0:s0 + step]
        r = (v >> 16) & 1
        r += 0x7FFF
        r += v
        r >>= 16
        out[s0:s0 + step] = r
    return out.reshape(np.shape(a))


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    b = np.ascontiguousarray(bits).reshape(-1)
    out = np.empty(b.size, np.uint32)
    step = 1 << 22
    for s0 in range(0, b.size, step):
        o = out[s0:s0 + step]
        o[:] = b[s0:s0 + step]
        o <<= 16
    return out.view(np.float32).reshape(np.shape(bits))


def _gelu(a: np.ndarray) -> np.ndarray:
    try:
        from scipy.special import erf
        e = erf(a / np.float32(np.sqrt(2.0))).astype(np.float32)
    except ImportError:  # pragma: no cover - scipy is in both images
        import torch
        e = torch.special.erf(torch.from_numpy(a) / float(np.sqrt(2.0))).numpy()
    return (np.float32(0.5) * a * (np.float32(1.0) + e)).astype(np.float32)


def _streams(seed: int):
    ss = np.random.SeedSequence(seed)
    return [np.random.default_rng(s) for s in ss.spawn(4)]


def draw_supports(C: int, R: int, k: int, support_pool: int, rng: np.random.Generator):
    """k distinct channels per expert from one random subset of support_pool channels."""
    if not (1 <= k <= support_pool <= C):
        raise ValueError("need 1 <= k <= support_pool <= C_in")
    pool = rng.choice(C, size=support_pool, replace=False)
    idx = np.empty((R, k), np.int32)
    for e in range(R):
        idx[e] = rng.choice(pool, size=k, replace=False)
    return idx


def cyclic_supports(C: int, R: int, k: int) -> np.ndarray:
    """Deterministic cyclic supports of Sec. 4.5 (0-based): S_e = {(e*k + j) mod C}."""
    e = np.arange(R, dtype=np.int64)[:, None]
    j = np.arange(k, dtype=np.int64)[None, :]
    return ((e * k + j) % C).astype(np.int32)


def make_x(cfg: LayerConfig, rng: np.random.Generator):
    """Post-activation input in cfg.layout; returns (float32 values, bf16 bits or None)."""
    a = rng.standard_normal((cfg.N, cfg.H, cfg.W, cfg.C_in), dtype=np.float32)
    if cfg.activation == "relu":
        np.maximum(a, np.float32(0.0), out=a)
    elif cfg.activation == "gelu":
        a = _gelu(a)
    else:
        raise ValueError(cfg.activation)
    if cfg.layout == "nchw":
        a = np.ascontiguousarray(a.transpose(0, 3, 1, 2))
    bits = None
    if cfg.dtype == "bf16":
        bits = bf16_bits(a)
        a = bf16_to_f32(bits)
    elif cfg.dtype != "f32":
        raise ValueError(cfg.dtype)
    return a, bits


def make_layer(cfg: LayerConfig, seed: int = 0) -> SyntheticLayer:
    rx, rs, rl, rg = _streams(seed)
    x, bits = make_x(cfg, rx)
    R, k = cfg.C_out, cfg.k
    sidx = draw_supports(cfg.C_in, R, k, cfg.support_pool, rs)
    slog = rl.standard_normal((R, k), dtype=np.float32)
    std = np.float32(1.0 / np.sqrt(k))
    W1 = (rg.standard_normal((k, k), dtype=np.float32) * std).astype(np.float32)
    w2 = (rg.standard_normal(k, dtype=np.float32) * std).astype(np.float32)
    if cfg.gate_bias_zero:
        b1 = np.zeros(k, np.float32)
        b2 = np.zeros(1, np.float32)
    else:
        b1 = (rg.standard_normal(k, dtype=np.float32) * std).astype(np.float32)
        b2 = (rg.standard_normal(1, dtype=np.float32) * std).astype(np.float32)
    return SyntheticLayer(cfg, x, bits, sidx, slog, W1, b1, w2, b2)


def make_dy(cfg: LayerConfig, seed: int = 0):
    """Upstream gradient dJ/dy of a scalar J, the shape, layout and dtype of y
    (C_out + 1 channels); returns (float32 values, bf16 bits or None)."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0x5EED]))
    shape = (cfg.N, cfg.H, cfg.W, cfg.C_out + 1)
    if cfg.layout == "nchw":
        shape = (cfg.N, cfg.C_out + 1, cfg.H, cfg.W)
    a = rng.standard_normal(shape, dtype=np.float32)
    bits = None
    if cfg.dtype == "bf16":
        bits = bf16_bits(a)
        a = bf16_to_f32(bits)
    return a, bits


def make_dynamic_x(cfg: LayerConfig, seed: int = 0, mean_std: float = 0.5,
                   grid: float | None = None):
    """Activations for the input-conditioned variant: act(N(mu[n, c], 1)) with per-example
    channel means mu ~ N(0, mean_std^2), so that the pooled descriptors (the router's input)
    differ between examples as real feature maps do. With `grid`, values are rounded to
    multiples of it (1/16: every partial sum of a pool is then exact in fp32). Returns
    (float32 values, bf16 bits or None) in cfg.layout."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0xD1]))
    mu = (rng.standard_normal((cfg.N, 1, 1, cfg.C_in)) * mean_std).astype(np.float32)
    a = rng.standard_normal((cfg.N, cfg.H, cfg.W, cfg.C_in), dtype=np.float32) + mu
    if cfg.activation == "relu":
        np.maximum(a, np.float32(0.0), out=a)
    else:
        a = _gelu(a)
    if grid is not None:
        a = (np.round(a / np.float32(grid)) * np.float32(grid)).astype(np.float32)
    if cfg.layout == "nchw":
        a = np.ascontiguousarray(a.transpose(0, 3, 1, 2))
    bits = None
    if cfg.dtype == "bf16":
        bits = bf16_bits(a)
        a = bf16_to_f32(bits)
    return a, bits


def make_router(cfg: LayerConfig, d: int, seed: int = 0):
    """Parameters of the rank-d router of Eq. (dynamic): the static routing matrix L ~ N(0, 1)
    [C_out, C_in], W_h ~ N(0, 1/C_in) [d, C_in], b_h ~ N(0, 0.01) [d], v_c ~ N(0, 1/d) [C_in, d],
    q_e ~ N(0, 4) [C_out, d] (so the offset is of the order of the logits' spread)."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0xD2]))
    R, C = cfg.C_out, cfg.C_in
    f = np.float32
    return {"L": rng.standard_normal((R, C), dtype=f),
            "Wh": (rng.standard_normal((d, C), dtype=f) / f(np.sqrt(C))).astype(f),
            "bh": (rng.standard_normal(d, dtype=f) * f(0.1)).astype(f),
            "V": (rng.standard_normal((C, d), dtype=f) / f(np.sqrt(d))).astype(f),
            "Q": (rng.standard_normal((R, d), dtype=f) * f(2.0)).astype(f)}


def x_to_layout(x: np.ndarray, src: str, dst: str) -> np.ndarray:
    if src == dst:
        return x
    if src == "nhwc" and dst == "nchw":
        return np.ascontiguousarray(x.transpose(0, 3, 1, 2))
    if src == "nchw" and dst == "nhwc":
        return np.ascontiguousarray(x.transpose(0, 2, 3, 1))
    raise ValueError((src, dst))
