"""Seeded inputs for the VLM's LLM prefill (Gemma-2B-shaped): configuration, weights and the
prefix token embeddings. Shapes and draws only; no arithmetic of the method."""

from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import numpy as np

from .inputs import _draw, round_to_bf16


@dataclass(frozen=True)
class LLMConfig:
    n_layers: int
    width: int          # W, residual width of the LLM
    n_heads: int        # H query heads; one shared KV head (the expert attends over it)
    head_dim: int       # D
    mlp_dim: int        # F, GeGLU hidden size
    rope_base: float = 10000.0      # 0 disables rotary position encoding
    rms_eps: float = 1e-6
    precision: str = "bf16"

    def with_(self, **kw) -> "LLMConfig":
        return replace(self, **kw)


# Gemma-2B-shaped LLM of pi0.5 (Tab. "Model architecture parameters of pi series VLA models":
# 18 layers, width 2048, 8 heads x 256); the GeGLU width 16384 is Gemma-2B's.
GEMMA2B = LLMConfig(n_layers=18, width=2048, n_heads=8, head_dim=256, mlp_dim=16384)

LLM_LAYER_WEIGHTS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")


def llm_weight_shapes(cfg: LLMConfig) -> dict:
    """Shape of every weight tensor; matrices are [out][in]."""
    W, H, D, F = cfg.width, cfg.n_heads, cfg.head_dim, cfg.mlp_dim
    return {
        "attn_norm": (W,), "wq": (H * D, W), "wk": (D, W), "wv": (D, W), "wo": (W, H * D),
        "mlp_norm": (W,), "w_gate": (F, W), "w_up": (F, W), "w_down": (W, F),
        "final_norm": (W,),
    }


def make_llm_weights(cfg: LLMConfig, seed: int, std: float = 0.02, norm_std: float = 0.1) -> dict:
    """{name: [array per layer]} for the layer tensors and {"final_norm": array}; fp32, the
    matrices bf16-representable in bf16 precision. Norm scales w enter as (1 + w)."""
    shapes = llm_weight_shapes(cfg)
    order = [(name, l) for l in range(cfg.n_layers) for name in LLM_LAYER_WEIGHTS] + [("final_norm", None)]
    bf16 = cfg.precision == "bf16"

    def one(j):
        name = order[j][0]
        rng = np.random.Generator(np.random.PCG64([seed, 104729, j]))
        shp = shapes[name]
        if len(shp) == 2:
            x = _draw(rng, shp, std)
            return round_to_bf16(x) if bf16 else x
        return _draw(rng, shp, norm_std)

    with ThreadPoolExecutor(max_workers=8) as ex:
        arrays = list(ex.map(one, range(len(order))))
    out = {name: [None] * cfg.n_layers for name in LLM_LAYER_WEIGHTS}
    for (name, l), a in zip(order, arrays):
        if l is None:
            out[name] = a
        else:
            out[name][l] = a
    return out


def make_prefix_embeddings(cfg: LLMConfig, seed: int, batch: int, prefix_len: int) -> np.ndarray:
    """Prefix token embeddings [B][P][W] (image and text tokens as the LLM receives them),
    N(0, 1), request b from its own generator; bf16-representable in bf16 precision."""
    out = np.empty((batch, prefix_len, cfg.width), np.float32)
    for b in range(batch):
        rng = np.random.Generator(np.random.PCG64([seed, 1299709, b]))
        out[b] = _draw(rng, (prefix_len, cfg.width), 1.0)
    return round_to_bf16(out) if cfg.precision == "bf16" else out
