"""Seeded inputs for the future correction module and its Q-Former state compressor (Sec. 4.1,
App. B): configuration, weight shapes, weights and the per-request inputs. Shapes and draws
only; no arithmetic of the method.

Draw order (fixed, part of the input recipe): tensor j of ``correction_weight_order(cfg)`` is
drawn from its own Generator(PCG64([seed, 15485863, j])); request b's inputs from
Generator(PCG64([seed, 32452843, b])), in the order VLM final-layer output, compressed state,
committed actions. Matrices and the learned query / position tables are N(0, std^2) (bf16-
representable in bf16 precision), biases N(0, bias_std^2), LayerNorm scales 1 + N(0,
norm_std^2), LayerNorm shifts N(0, bias_std^2).
"""

from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import numpy as np

from .inputs import _draw, round_to_bf16


@dataclass(frozen=True)
class CorrectionConfig:
    width: int          # module width = d_AE, the action expert's width (the correction item's)
    n_heads: int        # heads of every attention in the module
    head_dim: int       # width = n_heads * head_dim
    mlp_dim: int        # hidden size of every block's MLP
    d_vlm: int          # width of the VLM final-layer output the compressor reads
    n_items: int        # T', compressed tokens
    action_dim: int     # A
    max_delta: int      # longest committed-action sequence (rows of the position table)
    n_joint: int = 2    # Transformer blocks after the two branches are joined
    ln_eps: float = 1e-6
    precision: str = "bf16"

    def with_(self, **kw) -> "CorrectionConfig":
        return replace(self, **kw)


# pi0.5-sized module: d_AE = 1024 (the expert's width), d_VLM = 2048 (Gemma 2B), T' = 4
# (App. B), 8 heads x 128, MLP 2048; about 44M parameters (the paper quotes 40M, Sec. 4.1).
# max_delta = 50, one pi0.5 action chunk.
PI05_CORRECTION = CorrectionConfig(width=1024, n_heads=8, head_dim=128, mlp_dim=2048, d_vlm=2048,
                                   n_items=4, action_dim=32, max_delta=50)


def _attn_shapes(p: str, d: int, d_kv: int) -> dict:
    return {p + "wq": (d, d), p + "bq": (d,), p + "wk": (d, d_kv), p + "bk": (d,),
            p + "wv": (d, d_kv), p + "bv": (d,), p + "wo": (d, d), p + "bo": (d,)}


def _ln_shapes(p: str, d: int) -> dict:
    return {p + "_w": (d,), p + "_b": (d,)}


def _mlp_shapes(p: str, d: int, f: int) -> dict:
    return {p + "w1": (f, d), p + "b1": (f,), p + "w2": (d, f), p + "b2": (d,)}


def _block_shapes(p: str, d: int, f: int) -> dict:
    return {**_ln_shapes(p + "ln1", d), **_attn_shapes(p + "sa_", d, d),
            **_ln_shapes(p + "ln2", d), **_mlp_shapes(p + "mlp_", d, f)}


def correction_weight_shapes(cfg: CorrectionConfig) -> dict:
    """Every tensor, in draw order; matrices are [out][in].

    qf_*   Q-Former compressor: learned queries, self-attention, cross-attention into the VLM
           output (keys and values from width d_vlm), MLP, output LayerNorm.
    act_*  action branch: per-action MLP, position table, one Transformer block (ab_*).
    fuse_* projection of the joined branches; jb{i}_* the joint blocks; head_ln, corr_*,
           conf_* the two heads.
    """
    d, f, dv = cfg.width, cfg.mlp_dim, cfg.d_vlm
    s = {"qf_query": (cfg.n_items, d)}
    s.update(_ln_shapes("qf_ln1", d))
    s.update(_attn_shapes("qf_sa_", d, d))
    s.update(_ln_shapes("qf_ln2", d))
    s.update(_attn_shapes("qf_ca_", d, dv))
    s.update(_ln_shapes("qf_ln3", d))
    s.update(_mlp_shapes("qf_mlp_", d, f))
    s.update(_ln_shapes("qf_lnf", d))
    s.update({"act_w1": (d, cfg.action_dim), "act_b1": (d,), "act_w2": (d, d), "act_b2": (d,),
              "act_pos": (cfg.max_delta, d)})
    s.update(_block_shapes("ab_", d, f))
    s.update({"fuse_w": (d, 2 * d), "fuse_b": (d,)})
    for i in range(cfg.n_joint):
        s.update(_block_shapes(f"jb{i}_", d, f))
    s.update(_ln_shapes("head_ln", d))
    s.update({"corr_w": (d, d), "corr_b": (d,), "conf_w": (1, d), "conf_b": (1,)})
    return s


def correction_param_count(cfg: CorrectionConfig) -> int:
    return sum(int(np.prod(v)) for v in correction_weight_shapes(cfg).values())


def make_correction_weights(cfg: CorrectionConfig, seed: int, std: float = 0.02,
                            bias_std: float = 0.02, norm_std: float = 0.1) -> dict:
    """{name: fp32 array} for every tensor of ``correction_weight_shapes``."""
    shapes = correction_weight_shapes(cfg)
    names = list(shapes)
    bf16 = cfg.precision == "bf16"

    def one(j):
        name = names[j]
        rng = np.random.Generator(np.random.PCG64([seed, 15485863, j]))
        shp = shapes[name]
        if len(shp) == 2:
            x = _draw(rng, shp, std)
            return round_to_bf16(x) if bf16 else x
        if name.endswith("_w") and "ln" in name:
            return (np.float32(1.0) + _draw(rng, shp, norm_std)).astype(np.float32)
        return _draw(rng, shp, bias_std)

    with ThreadPoolExecutor(max_workers=8) as ex:
        arrays = list(ex.map(one, range(len(names))))
    return dict(zip(names, arrays))


def make_correction_inputs(cfg: CorrectionConfig, seed: int, batch: int, n_vlm_tokens: int,
                           delta: int, first_request: int = 0) -> dict:
    """Per-request inputs: the VLM final-layer output h_vlm [B][T][d_vlm] (bf16-representable in
    bf16 precision, N(0, 1)), a compressed state [B][T'][width] N(0, 1) (the state buffer's
    content when the VLM was skipped) and the committed actions [B][delta][A] N(0, 1)."""
    hv = np.empty((batch, n_vlm_tokens, cfg.d_vlm), np.float32)
    hc = np.empty((batch, cfg.n_items, cfg.width), np.float32)
    acts = np.empty((batch, delta, cfg.action_dim), np.float32)
    for b in range(batch):
        rng = np.random.Generator(np.random.PCG64([seed, 32452843, first_request + b]))
        hv[b] = _draw(rng, (n_vlm_tokens, cfg.d_vlm), 1.0)
        hc[b] = _draw(rng, (cfg.n_items, cfg.width), 1.0)
        acts[b] = _draw(rng, (delta, cfg.action_dim), 1.0)
    if cfg.precision == "bf16":
        hv = round_to_bf16(hv)
    return {"h_vlm": hv, "h_c": hc, "actions": acts}
