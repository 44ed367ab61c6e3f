"""CPU oracle for the VLM's LLM prefill, the step that produces the per-layer KV cache the action
expert attends over (fp64, numpy).

TEST INFRASTRUCTURE ONLY. Only the tests, the smoke check and the bench's CPU legs may import
it; the library never does, and it shares no code with the CUDA path.

What the paper fixes (App. A "Model Architecture of pi series Models", Tab. "Model architecture
parameters of pi series VLA models", Sec. 4.3): the LLM (Gemma 2B: 18 layers, width 2048,
8 attention heads of dimension 256) processes the concatenated visual and language tokens and
provides the KV cache of each layer, which the matching expert layer concatenates with its own
keys and values. Everything else is a reading (numbered after the expert's R1..R15):
  R16 one KV head of width D shared by the H query heads (the expert's attention consumes one
      KV head of width 256 per layer).
  R17 Gemma pre-norm block without biases: h += Wo attn(u), u = rms(h) (1 + a); then
      h += Wd (gelu_tanh(Wg u) * (Wu u)), u = rms(h) (1 + m); GeGLU width 16384 (Gemma 2B).
  R18 rotary coding (rotate-half, base rope_base) of q and k at positions 0..P-1; the cached K
      is the rotated one (the expert uses the prefix K as given, R6).
  R19 every prefix token sees every prefix token (image and language tokens form one
      bidirectional block).
  R20 layer l's KV comes from layer l's input stream; the final-layer output is
      rms(h) (1 + final_norm), the VLM state the correction module compresses.
"""

from __future__ import annotations

import numpy as np

from .expert import F64, attention, gelu_tanh, rms_modulate, rope


def llm_prefill(x: np.ndarray, w: dict, cfg, return_output: bool = False):
    """KV cache K, V [L][P][D] of one request's prefix embeddings x [P][W] (App. A).

    With return_output, also the final-layer output [P][W] (R20)."""
    P, W = x.shape
    L, H, D = cfg.n_layers, cfg.n_heads, cfg.head_dim
    h = x.astype(F64)
    pos = np.arange(P)
    visible = np.ones((P, P), dtype=bool)                          # R19
    K = np.empty((L, P, D), dtype=F64)
    V = np.empty((L, P, D), dtype=F64)
    for l in range(L):
        u = rms_modulate(h, w["attn_norm"][l], 0.0, cfg.rms_eps)   # R17
        q = (u @ w["wq"][l].T).reshape(P, H, D)
        k = u @ w["wk"][l].T                                       # R16
        v = u @ w["wv"][l].T
        q = rope(q, pos, cfg.rope_base)                            # R18
        k = rope(k, pos, cfg.rope_base)
        K[l], V[l] = k, v                                          # R20
        o = attention(q, k, v, visible).reshape(P, H * D)
        h = h + o @ w["wo"][l].T
        u = rms_modulate(h, w["mlp_norm"][l], 0.0, cfg.rms_eps)
        h = h + (gelu_tanh(u @ w["w_gate"][l].T) * (u @ w["w_up"][l].T)) @ w["w_down"][l].T
    if return_output:
        return K, V, rms_modulate(h, w["final_norm"], 0.0, cfg.rms_eps)
    return K, V


def to_f64_llm(w: dict) -> dict:
    return {k: ([np.asarray(a, F64) for a in v] if isinstance(v, list) else np.asarray(v, F64))
            for k, v in w.items()}


def prefill_batch(x: np.ndarray, w: dict, cfg):
    """Each request b independently: x [B][P][W] -> K, V [L][B][P][D] and the outputs [B][P][W]."""
    w64 = to_f64_llm(w)
    res = [llm_prefill(x[b], w64, cfg, return_output=True) for b in range(x.shape[0])]
    K = np.stack([r[0] for r in res], axis=1)
    V = np.stack([r[1] for r in res], axis=1)
    return K, V, np.stack([r[2] for r in res])
