"""Seeded synthetic workloads for the rolling action-expert step.

This module only *draws* inputs: expert shapes, random-init weights, VLM prefix
K/V, Fast-Observation-Pathway tokens, slot flow times, context offsets and
per-robot seeds.  It contains none of the step's arithmetic, so that both the
fp64 CPU oracle (``oracle/``) and the CUDA library can be fed the very same
arrays without sharing any computation.

Recipe (the paper runs on LIBERO / RoboTwin / DOM / real robots with released
checkpoints, none of which exist here; these seeded tensors stand in for them):

* weights and biases ~ N(0, 0.02), every parameter, one numpy PCG64 stream per
  named tensor (seed derived from the weight seed and the tensor's name);
* prefix K/V ~ N(0, 1), [L, B, Hkv, P, hd], robot b drawn from seed ``base+b``;
* FOP tokens ~ N(0, 1), [B, F, D], robot b from seed ``base+b``;
* slot flow times t_j = (j+1)/H (t = 1 is pure noise, j = 0 is the slot that is
  released next);
* in bf16 mode every weight, prefix and FOP value is rounded to the nearest
  bf16 (ties to even) and kept as float32, so both sides read identical values.
"""
from __future__ import annotations

import dataclasses
import hashlib
from dataclasses import dataclass

import numpy as np

__all__ = [
    "ExpertConfig", "PRESETS", "SWEEP", "round_bf16", "make_weights", "weight_names",
    "make_context", "make_fop", "staggered_times", "robot_seeds", "make_delta",
]


@dataclass(frozen=True)
class ExpertConfig:
    """Shape of the action expert and of one rolling step.

    Field names follow the build's notation: H slots (the paper's K, with h = 1
    action per slot), A action dim, D width, L layers, Hq / Hkv query / KV heads,
    hd head dim, Fm MLP hidden width, P prefix tokens, F FOP tokens, B robots.
    """
    layers: int
    width: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    mlp_dim: int
    slots: int
    action_dim: int
    prefix: int
    fop_tokens: int
    batch: int
    dtype: str  # "fp32" or "bf16"
    # 0: FOP tokens are extra keys / values of every layer's self-attention;
    # k > 0: they enter layers k-1, 2k-1, ... through gated cross-attention
    # adapters instead (and are not keys of the self-attention)
    fop_adapter_every: int = 0
    per_robot_times: int = 0     # 1: slot times [B, H], one schedule per robot

    @property
    def n_adapters(self) -> int:
        return self.layers // self.fop_adapter_every if self.fop_adapter_every else 0

    @property
    def n_qkv(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    @property
    def q_dim(self) -> int:
        return self.n_q_heads * self.head_dim

    @property
    def mod_dim(self) -> int:
        """Columns of the modulation Dense: (scale1, shift1, scale2, shift2) per
        layer, then (scale, shift) of the final norm."""
        return 4 * self.layers * self.width + 2 * self.width

    def replace(self, **kw) -> "ExpertConfig":
        return dataclasses.replace(self, **kw)

    def param_count(self) -> int:
        D, L = self.width, self.layers
        layer = D * self.n_qkv + self.q_dim * D + 3 * D * self.mlp_dim + D
        cond = 2 * (2 * D * D + 2 * D)
        return (L * layer + cond + D * self.mod_dim + self.mod_dim
                + self.action_dim * D + D + D * self.action_dim + self.action_dim)


_PI05 = dict(layers=18, width=1024, n_q_heads=8, n_kv_heads=1, head_dim=256, mlp_dim=4096,
             slots=50, action_dim=32, prefix=816, fop_tokens=16)

PRESETS: dict[str, ExpertConfig] = {
    # tiny expert, fp32, one robot
    "tiny_fp32_b1": ExpertConfig(layers=2, width=256, n_q_heads=4, n_kv_heads=1, head_dim=64,
                                 mlp_dim=1024, slots=10, action_dim=7, prefix=64, fop_tokens=4,
                                 batch=1, dtype="fp32"),
    # pi0.5-style expert shape, bf16, one robot (the latency workload)
    "pi05_bf16_b1": ExpertConfig(**_PI05, batch=1, dtype="bf16"),
    # same expert, 64 independent robots (the throughput workload)
    "pi05_bf16_b64": ExpertConfig(**_PI05, batch=64, dtype="bf16"),
    # wider GQA expert, eight robots
    "wide_bf16_b8": ExpertConfig(layers=24, width=1024, n_q_heads=16, n_kv_heads=4, head_dim=64,
                                 mlp_dim=4096, slots=30, action_dim=20, prefix=512,
                                 fop_tokens=32, batch=8, dtype="bf16"),
}

# Stress grid over the pi0.5-shaped expert: batch x prefix length x slots.
SWEEP: list[ExpertConfig] = [
    PRESETS["pi05_bf16_b1"].replace(batch=b, prefix=p, slots=h)
    for b in (1, 16, 64, 256) for p in (256, 816, 2048) for h in (16, 50)
]


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), returned as
    float32.  Inputs here are finite."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(x.shape)


def _stream(seed: int, name: str) -> np.random.Generator:
    h = hashlib.sha256(f"{seed}:{name}".encode()).digest()
    return np.random.default_rng(int.from_bytes(h[:8], "little"))


def weight_names(cfg: ExpertConfig) -> dict[str, tuple[int, ...]]:
    """Named parameters in math layout (y = x @ W + b, W is [in, out]).

    Per-layer tensors are stacked on a leading L axis.  The QKV columns are
    [Q heads | K heads | V heads], each head ``hd`` wide.
    """
    D, L, A = cfg.width, cfg.layers, cfg.action_dim
    return {
        "t_w1": (D, D), "t_b1": (D,), "t_w2": (D, D), "t_b2": (D,),
        "d_w1": (D, D), "d_b1": (D,), "d_w2": (D, D), "d_b2": (D,),
        "mod_w": (D, cfg.mod_dim), "mod_b": (cfg.mod_dim,),
        "in_w": (A, D), "in_b": (D,),
        "fop_gamma": (L, D),
        "w_qkv": (L, D, cfg.n_qkv),
        "w_o": (L, cfg.q_dim, D),
        "w_gate": (L, D, cfg.mlp_dim),
        "w_up": (L, D, cfg.mlp_dim),
        "w_down": (L, cfg.mlp_dim, D),
        "out_w": (D, A), "out_b": (A,),
        **({} if not cfg.n_adapters else {
            "a_gamma": (cfg.n_adapters, D), "a_zgamma": (cfg.n_adapters, D),
            "a_wq": (cfg.n_adapters, D, cfg.q_dim), "a_wkv": (cfg.n_adapters, D, 2 * cfg.n_kv_heads * cfg.head_dim),
            "a_wo": (cfg.n_adapters, cfg.q_dim, D), "a_gate": (cfg.n_adapters,)}),
    }


def make_weights(cfg: ExpertConfig, seed: int = 0, std: float = 0.02) -> dict[str, np.ndarray]:
    """Every parameter ~ N(0, std) as float32 (bf16-representable in bf16 mode)."""
    out = {}
    for name, shape in weight_names(cfg).items():
        w = _stream(seed, name).standard_normal(shape, dtype=np.float32) * np.float32(std)
        out[name] = round_bf16(w) if cfg.dtype == "bf16" else w
    return out


def make_context(cfg: ExpertConfig, base_seed: int, batch: int | None = None,
                 prefix_len: int | None = None) -> tuple[np.ndarray, np.ndarray]:
    """Prefix K and V ~ N(0,1), each [L, B, Hkv, prefix_len, hd] float32."""
    B = cfg.batch if batch is None else batch
    P = cfg.prefix if prefix_len is None else prefix_len
    shp = (cfg.layers, cfg.n_kv_heads, P, cfg.head_dim)
    k = np.empty((cfg.layers, B, cfg.n_kv_heads, P, cfg.head_dim), np.float32)
    v = np.empty_like(k)
    for b in range(B):
        g = _stream(base_seed + b, "prefix_kv")
        k[:, b] = g.standard_normal(shp, dtype=np.float32)
        v[:, b] = g.standard_normal(shp, dtype=np.float32)
    if cfg.dtype == "bf16":
        k, v = round_bf16(k), round_bf16(v)
    return k, v


def make_fop(cfg: ExpertConfig, base_seed: int, batch: int | None = None) -> np.ndarray:
    """Fast-Observation-Pathway tokens ~ N(0,1), [B, F, D] float32."""
    B = cfg.batch if batch is None else batch
    z = np.stack([_stream(base_seed + b, "fop").standard_normal(
        (cfg.fop_tokens, cfg.width), dtype=np.float32) for b in range(B)]) if B else \
        np.zeros((0, cfg.fop_tokens, cfg.width), np.float32)
    return round_bf16(z) if cfg.dtype == "bf16" else z


def staggered_times(H: int) -> np.ndarray:
    """Flow times t_j = (j+1)/H of the H slots, as float32."""
    return ((np.arange(H, dtype=np.float64) + 1.0) / H).astype(np.float32)


def robot_seeds(base: int, B: int) -> np.ndarray:
    """Per-robot noise seeds base + b as uint64."""
    return (np.uint64(base) + np.arange(B, dtype=np.uint64)).astype(np.uint64)


def make_delta(B: int, age_steps, H: int, bias: float = 0.0) -> np.ndarray:
    """Context-age offsets delta_b = p_b / H + bias as float32, one per robot."""
    p = np.broadcast_to(np.asarray(age_steps, dtype=np.float64), (B,))
    return (p / H + bias).astype(np.float32)
