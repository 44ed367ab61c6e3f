"""Shapes and seeded draws for the action expert's inputs.

Sizes follow the pi0.5 action expert (Tab. "Model architecture parameters of pi series VLA
models": 18 layers, width 1024, 8 heads x 256) and its LLM prefix (Gemma 2B, 256 tokens per
224x224 image at patch 14). Every tensor is drawn from numpy's PCG64 in a fixed order, so a
seed fixes every value bit for bit on any machine.

Draw order (fixed, part of the input recipe):
  weights: tensor j in the order "global tensors in ``GLOBAL_WEIGHTS`` order, then for each
           layer the tensors in ``LAYER_WEIGHTS`` order" is drawn from its own
           Generator(PCG64([seed, j])) (independent streams, so tensors are drawn in parallel).
  request b: Generator(PCG64([seed, b])); prefix K for every layer, prefix V for every layer,
           then the state vector, then the action noise.
Weight matrices are N(0, std^2); biases N(0, bias_std^2) (the three modulation biases can be
given their own std to drive the adaptive-norm gates to O(1)); prefix K/V, state and noise
are N(0, 1). In bf16 precision every weight matrix and the prefix K/V are rounded to the
nearest bf16 value (ties to even) here, and both the oracle and the CUDA path consume those
exact values; biases, state and noise stay fp32.
"""

from __future__ import annotations

from dataclasses import dataclass, replace

from concurrent.futures import ThreadPoolExecutor

import numpy as np


@dataclass(frozen=True)
class ExpertConfig:
    n_layers: int
    width: int          # W, residual width of the expert
    n_heads: int        # H query heads; the expert has a single shared KV head
    head_dim: int       # D
    mlp_dim: int        # F, GeGLU hidden size
    action_dim: int     # A
    state_dim: int      # S_d (continuous state token input size)
    time_dim: int       # d_t, sinusoidal time-embedding size
    rope_base: float = 10000.0      # 0 disables rotary position encoding of the suffix
    rms_eps: float = 1e-6
    t_min_period: float = 4e-3
    t_max_period: float = 4.0
    precision: str = "bf16"         # "bf16" (bf16 weights) or "fp32"

    def with_(self, **kw) -> "ExpertConfig":
        return replace(self, **kw)


# Tiny fp32 expert: 2 layers, width 256, 4 heads x 64, GeGLU 1024, 64-dim time embedding.
TINY = ExpertConfig(n_layers=2, width=256, n_heads=4, head_dim=64, mlp_dim=1024,
                    action_dim=7, state_dim=7, time_dim=64, precision="fp32")

# pi0.5-shaped action expert (Gemma-300M-like): 18 x (1024, 8 x 256, GeGLU 4096), 32-dim actions.
PI05 = ExpertConfig(n_layers=18, width=1024, n_heads=8, head_dim=256, mlp_dim=4096,
                    action_dim=32, state_dim=32, time_dim=1024, precision="bf16")

GLOBAL_WEIGHTS = (
    "state_in_w", "state_in_b", "action_in_w", "action_in_b",
    "action_out_w", "action_out_b",
    "time_mlp_in_w", "time_mlp_in_b", "time_mlp_out_w", "time_mlp_out_b",
    "final_mod_w", "final_mod_b",
)

LAYER_WEIGHTS = (
    "wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down",
    "attn_mod_w", "attn_mod_b", "mlp_mod_w", "mlp_mod_b",
)

_MOD_BIASES = ("attn_mod_b", "mlp_mod_b", "final_mod_b")


def weight_shapes(cfg: ExpertConfig) -> dict:
    """Shape of every weight tensor; matrices are [out][in] (nn.Linear layout)."""
    W, H, D, F = cfg.width, cfg.n_heads, cfg.head_dim, cfg.mlp_dim
    A, Sd, dt = cfg.action_dim, cfg.state_dim, cfg.time_dim
    return {
        "state_in_w": (W, Sd), "state_in_b": (W,),
        "action_in_w": (W, A), "action_in_b": (W,),
        "action_out_w": (A, W), "action_out_b": (A,),
        "time_mlp_in_w": (W, dt), "time_mlp_in_b": (W,),
        "time_mlp_out_w": (W, W), "time_mlp_out_b": (W,),
        "final_mod_w": (2 * W, W), "final_mod_b": (2 * W,),
        "wq": (H * D, W), "wk": (D, W), "wv": (D, W), "wo": (W, H * D),
        "w_gate": (F, W), "w_up": (F, W), "w_down": (W, F),
        "attn_mod_w": (3 * W, W), "attn_mod_b": (3 * W,),
        "mlp_mod_w": (3 * W, W), "mlp_mod_b": (3 * W,),
    }


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """fp32 array whose values are ``a`` rounded to bf16 (nearest, ties to even); finite input."""
    u = np.array(a, dtype=np.float32, copy=True).view(np.uint32)
    u += np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    u &= np.uint32(0xFFFF0000)
    return u.view(np.float32)


def _draw(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    x = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    return x


def make_weights(cfg: ExpertConfig, seed: int, std: float = 0.02, bias_std: float = 0.02,
                 mod_bias_std: float | None = None) -> dict:
    """All expert weights as fp32 numpy arrays.

    Returns ``{name: array}`` for the global tensors and ``{name: [array per layer]}`` for the
    per-layer tensors. In bf16 precision the matrices hold bf16-representable values.
    """
    if mod_bias_std is None:
        mod_bias_std = bias_std
    shapes = weight_shapes(cfg)
    bf16 = cfg.precision == "bf16"
    order = [(name, None) for name in GLOBAL_WEIGHTS] + [
        (name, l) for l in range(cfg.n_layers) for name in LAYER_WEIGHTS]

    def one(j):
        name = order[j][0]
        rng = np.random.Generator(np.random.PCG64([seed, j]))
        shp = shapes[name]
        if len(shp) == 2:
            x = _draw(rng, shp, std)
            return round_to_bf16(x) if bf16 else x
        return _draw(rng, shp, mod_bias_std if name in _MOD_BIASES else bias_std)

    with ThreadPoolExecutor(max_workers=8) as ex:
        arrays = list(ex.map(one, range(len(order))))
    out = {}
    per_layer = {name: [None] * cfg.n_layers for name in LAYER_WEIGHTS}
    for (name, l), a in zip(order, arrays):
        if l is None:
            out[name] = a
        else:
            per_layer[name][l] = a
    out.update(per_layer)
    return out


def make_requests(cfg: ExpertConfig, seed: int, batch: int, prefix_len: int, chunk: int,
                  first_request: int = 0) -> dict:
    """Per-request inputs: prefix K/V [L][B][P][D], state [B][S_d], noise [B][C][A] (fp32).

    Request ``b`` (0-based, offset by ``first_request``) is drawn from its own generator, so a
    batch is the concatenation of independently seeded single requests.
    """
    L, D = cfg.n_layers, cfg.head_dim
    bf16 = cfg.precision == "bf16"
    K = np.empty((L, batch, prefix_len, D), np.float32)
    V = np.empty((L, batch, prefix_len, D), np.float32)
    state = np.empty((batch, cfg.state_dim), np.float32)
    noise = np.empty((batch, chunk, cfg.action_dim), np.float32)
    def one(b):
        rng = np.random.Generator(np.random.PCG64([seed, first_request + b]))
        for l in range(L):
            K[l, b] = _draw(rng, (prefix_len, D), 1.0)
        for l in range(L):
            V[l, b] = _draw(rng, (prefix_len, D), 1.0)
        state[b] = _draw(rng, (cfg.state_dim,), 1.0)
        noise[b] = _draw(rng, (chunk, cfg.action_dim), 1.0)

    with ThreadPoolExecutor(max_workers=8) as ex:
        list(ex.map(one, range(batch)))
    if bf16:
        K = round_to_bf16(K)
        V = round_to_bf16(V)
    return {"prefix_k": K, "prefix_v": V, "state": state, "noise": noise}


def make_correction(cfg: ExpertConfig, seed: int, batch: int, num_items: int,
                    first_request: int = 0, std: float = 1.0) -> np.ndarray:
    """Correction items [B][T'][width] fp32 (the compressed future VLM state given to the
    expert), request ``b`` from its own generator, separate from ``make_requests``' streams."""
    out = np.empty((batch, num_items, cfg.width), np.float32)
    for b in range(batch):
        rng = np.random.Generator(np.random.PCG64([seed, 7919, first_request + b]))
        out[b] = _draw(rng, (num_items, cfg.width), std)
    return out
