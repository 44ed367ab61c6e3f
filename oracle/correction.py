"""CPU oracle for the future correction module and its Q-Former state compressor (fp64, numpy).

TEST INFRASTRUCTURE ONLY. Only the tests, the smoke check and the bench's CPU legs may import
it; the library never does, and it shares no code with the CUDA path.

What the paper fixes (Sec. 4.1 "Foresight-Aligned Asynchronous Correction", App. B
"Architecture of Future Correction Module", Eq. 2, App. C Alg. 1): a compressor turns the VLM's
final-layer output [T][d_VLM] into T' = 4 tokens of width d_AE with one Q-Former block; the
module takes that compressed state and the committed actions a_t .. a_{t+Delta-1}, runs the
actions through an MLP and one Transformer block and keeps the last token, joins the two
branches, projects them, runs two more Transformer blocks, and ends in a correction head (the
predicted compressed state at t + Delta) and a confidence head (one scalar, trained toward
-L_predict by Eq. 2). About 40M parameters. Everything else is a reading (numbered after the
prefill's R16..R20):
  R21 the module's width is d_AE (the compressed state is the expert's correction item, R15);
      every attention has n_heads heads of head_dim with biased q/k/v/o projections, the
      1/sqrt(head_dim) scale and every key visible.
  R22 Transformer block = pre-LayerNorm: x += attn(LN1 x); x += MLP(LN2 x). LayerNorm is
      (x - mean) / sqrt(var + eps) * w + b with the biased variance.
  R23 MLP = W2 gelu_tanh(W1 x + b1) + b2 (the tanh GELU of R8).
  R24 Q-Former block: T' learned queries; self-attention among them, cross-attention from them
      into the VLM output (keys and values projected from d_VLM; the VLM tokens get no norm and
      no position code), MLP, each pre-LN with a residual; an output LayerNorm.
  R25 action branch: per-action MLP A -> d -> d, plus row k of a learned position table for
      action k, one Transformer block over the Delta tokens, its output at the last action.
      (After one block the last token's output is the same under a causal or a full mask.)
  R26 join: the action summary is appended to each compressed token feature-wise ([h_j ; s],
      width 2d) and projected to d; the joint blocks run over the T' tokens with no position
      table (the compressor's queries already tell the tokens apart).
  R27 heads: one shared LayerNorm; correction head = per-token linear map (the state itself,
      not a change to the input); confidence = linear map of the token mean, unsquashed.
  R28 Alg. 1: the compressor runs on each fresh VLM output; the state buffer holds compressed
      states, so when the VLM is skipped the last prediction is fed back in.
"""

from __future__ import annotations

import numpy as np

from .expert import F64, gelu_tanh


def layer_norm(x: np.ndarray, w: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    """R22: row-wise LayerNorm with the biased variance."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * w + b


def multi_head_attention(xq: np.ndarray, xkv: np.ndarray, w: dict, p: str, cfg) -> np.ndarray:
    """R21: queries from xq [n][d], keys and values from xkv [m][d_kv]; every key visible."""
    n, m, H, Dh = xq.shape[0], xkv.shape[0], cfg.n_heads, cfg.head_dim
    q = (xq @ w[p + "wq"].T + w[p + "bq"]).reshape(n, H, Dh)
    k = (xkv @ w[p + "wk"].T + w[p + "bk"]).reshape(m, H, Dh)
    v = (xkv @ w[p + "wv"].T + w[p + "bv"]).reshape(m, H, Dh)
    scores = np.einsum("ihd,jhd->hij", q, k) / np.sqrt(F64(Dh))
    scores = scores - scores.max(axis=-1, keepdims=True)
    pr = np.exp(scores)
    pr = pr / pr.sum(axis=-1, keepdims=True)
    o = np.einsum("hij,jhd->ihd", pr, v).reshape(n, H * Dh)
    return o @ w[p + "wo"].T + w[p + "bo"]


def mlp(x: np.ndarray, w: dict, p: str) -> np.ndarray:
    """R23."""
    return gelu_tanh(x @ w[p + "w1"].T + w[p + "b1"]) @ w[p + "w2"].T + w[p + "b2"]


def transformer_block(x: np.ndarray, w: dict, p: str, cfg) -> np.ndarray:
    """R22: pre-LN self-attention then MLP, each with a residual."""
    u = layer_norm(x, w[p + "ln1_w"], w[p + "ln1_b"], cfg.ln_eps)
    x = x + multi_head_attention(u, u, w, p + "sa_", cfg)
    u = layer_norm(x, w[p + "ln2_w"], w[p + "ln2_b"], cfg.ln_eps)
    return x + mlp(u, w, p + "mlp_")


def qformer_compress(h_vlm: np.ndarray, w: dict, cfg) -> np.ndarray:
    """App. B, R24: the VLM final-layer output [T][d_VLM] -> compressed state [T'][d_AE]."""
    x = w["qf_query"].copy()
    u = layer_norm(x, w["qf_ln1_w"], w["qf_ln1_b"], cfg.ln_eps)
    x = x + multi_head_attention(u, u, w, "qf_sa_", cfg)
    u = layer_norm(x, w["qf_ln2_w"], w["qf_ln2_b"], cfg.ln_eps)
    x = x + multi_head_attention(u, h_vlm, w, "qf_ca_", cfg)
    u = layer_norm(x, w["qf_ln3_w"], w["qf_ln3_b"], cfg.ln_eps)
    x = x + mlp(u, w, "qf_mlp_")
    return layer_norm(x, w["qf_lnf_w"], w["qf_lnf_b"], cfg.ln_eps)


def action_summary(actions: np.ndarray, w: dict, cfg) -> np.ndarray:
    """App. B, R25: committed actions [Delta][A] -> the last token's state [d]."""
    n = actions.shape[0]
    if not 1 <= n <= cfg.max_delta:
        raise ValueError(f"need 1..{cfg.max_delta} committed actions, got {n}")
    x = gelu_tanh(actions @ w["act_w1"].T + w["act_b1"]) @ w["act_w2"].T + w["act_b2"]
    x = x + w["act_pos"][:n]
    x = transformer_block(x, w, "ab_", cfg)
    return x[n - 1]


def future_correction(h_c: np.ndarray, actions: np.ndarray, w: dict, cfg):
    """App. B, R26, R27: f_corr(compressed state [T'][d], actions [Delta][A]) ->
    (predicted compressed state at t + Delta [T'][d], confidence)."""
    s = action_summary(actions, w, cfg)
    joined = np.concatenate([h_c, np.broadcast_to(s, h_c.shape)], axis=-1)
    x = joined @ w["fuse_w"].T + w["fuse_b"]
    for i in range(cfg.n_joint):
        x = transformer_block(x, w, f"jb{i}_", cfg)
    u = layer_norm(x, w["head_ln_w"], w["head_ln_b"], cfg.ln_eps)
    h_future = u @ w["corr_w"].T + w["corr_b"]
    confidence = float(w["conf_w"][0] @ u.mean(axis=0) + w["conf_b"][0])
    return h_future, confidence


def correct_from_vlm(h_vlm: np.ndarray, actions: np.ndarray, w: dict, cfg):
    """R28, the VLM branch of Alg. 1: compress a fresh VLM output, then predict ahead."""
    return future_correction(qformer_compress(h_vlm, w, cfg), actions, w, cfg)


def to_f64_corr(w: dict) -> dict:
    return {k: np.asarray(v, F64) for k, v in w.items()}


def compress_batch(h_vlm: np.ndarray, w: dict, cfg) -> np.ndarray:
    """Each request independently: [B][T][d_VLM] -> [B][T'][d]."""
    w64 = to_f64_corr(w)
    return np.stack([qformer_compress(np.asarray(h, F64), w64, cfg) for h in h_vlm])


def correction_batch(h_c: np.ndarray, actions: np.ndarray, w: dict, cfg):
    """Each request independently: [B][T'][d], [B][Delta][A] -> ([B][T'][d], [B])."""
    w64 = to_f64_corr(w)
    res = [future_correction(np.asarray(h_c[b], F64), np.asarray(actions[b], F64), w64, cfg)
           for b in range(h_c.shape[0])]
    return np.stack([r[0] for r in res]), np.array([r[1] for r in res], F64)
