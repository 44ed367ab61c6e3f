"""CPU oracle for the action expert's flow-matching denoise (fp64, numpy).

TEST INFRASTRUCTURE ONLY. This module defines what the denoise computes, slowly and plainly,
so that the CUDA path can be checked against it. Only the tests, the smoke check and the
bench's CPU-baseline leg may import it; the library never does, and it shares no code with
the CUDA path (the seeded input generator in ``synth`` is the only common module).

What the paper fixes (App. A "Model Architecture of pi series Models", Tab. "Model
architecture parameters of pi series VLA models", Sec. 4.3 "System Design"):
  * the action expert is a DiT whose queries come from the action-noise tokens and whose keys
    and values are the matching LLM layer's KV cache concatenated with those tokens;
  * 18 layers, width 1024, 8 attention heads of dimension 256;
  * flow matching refines noise into an action chunk over a fixed number of steps (10).
Everything else is a reading, numbered R1..R15 where it is used below:
  R1  time runs t_k = k/N, k = 0..N-1, with step delta = 1/N and x_{k+1} = x_k + delta * v.
  R2  sinusoidal time embedding, half sin / half cos, periods geometric from t_min_period to
      t_max_period.
  R3  time MLP: c = swish(W2 swish(W1 e + b1) + b2).
  R4  one continuous state token (linear projection) followed by the C action tokens.
  R5  adaptive RMSNorm: u = h / sqrt(mean(h^2) + eps) * (1 + sigma) + beta, with (sigma,
      beta, gamma) = split3(M c + m) per sublayer; gamma gates the sublayer output before
      the residual add; the final norm has (sigma, beta) only.
  R6  rotary position encoding (rotate-half, base rope_base) of suffix q and k at positions
      P + i; the prefix K is used as given. rope_base == 0 disables it.
  R7  attention scale 1/sqrt(D); the state row sees the prefix and itself, action rows see
      every prefix and suffix key; one KV head shared by all query heads.
  R8  GeGLU with tanh-approximated GELU.
  R9  velocity read from the action rows only.
  R10 requests in a batch are independent.
  R13 the Gemma projections (q, k, v, o, gate, up, down) carry no bias.
  R15 correction items (Sec. 4.1 "Foresight-Aligned Asynchronous Correction", App. B): the T'
      predicted compressed VLM states (width d_AE, the expert's width) given to the action
      expert enter it as context tokens right after the state token, taken as the residual
      stream's input row unchanged (no projection, d_AE = width). The state and context rows
      see the prefix and each other, action rows see every key, and the velocity is read from
      the action rows. With T' = 0 this is the plain expert.
"""

from __future__ import annotations

import numpy as np

F64 = np.float64


def sinusoidal_time_embedding(t: float, dim: int, min_period: float, max_period: float):
    """R2: [sin(2 pi t / p_i) ..., cos(2 pi t / p_i) ...], p_i geometric in i over half = dim/2.

    Flow time t enters the expert only through this embedding (App. A, flow matching).
    """
    half = dim // 2
    frac = np.arange(half, dtype=F64) / (half - 1)
    period = min_period * (max_period / min_period) ** frac
    theta = 2.0 * np.pi * F64(t) / period
    return np.concatenate([np.sin(theta), np.cos(theta)])


def swish(z):
    return z / (1.0 + np.exp(-z))


def time_conditioning(t: float, w: dict, cfg) -> np.ndarray:
    """R3: conditioning vector c [W] for flow time t."""
    e = sinusoidal_time_embedding(t, cfg.time_dim, cfg.t_min_period, cfg.t_max_period)
    c1 = swish(w["time_mlp_in_w"] @ e + w["time_mlp_in_b"])
    return swish(w["time_mlp_out_w"] @ c1 + w["time_mlp_out_b"])


def rms_modulate(h: np.ndarray, sigma: np.ndarray, beta: np.ndarray, eps: float):
    """R5: row-wise RMS normalisation followed by the time-conditioned scale and shift."""
    r = h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + eps)
    return r * (1.0 + sigma) + beta


def rope(x: np.ndarray, positions: np.ndarray, base: float) -> np.ndarray:
    """R6: rotate-half rotary encoding of x [n][..][D] at integer positions [n]."""
    if base == 0:
        return x
    D = x.shape[-1]
    half = D // 2
    omega = base ** (-2.0 * np.arange(half, dtype=F64) / D)
    ang = positions.astype(F64)[:, None] * omega[None, :]          # [n][half]
    shape = (x.shape[0],) + (1,) * (x.ndim - 2) + (half,)
    cos, sin = np.cos(ang).reshape(shape), np.sin(ang).reshape(shape)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * cos - b * sin, b * cos + a * sin], axis=-1)


def suffix_mask(prefix_len: int, suffix_len: int, n_ctx: int = 1) -> np.ndarray:
    """R7, R15: visible[i][n] for suffix row i and key n in [prefix; suffix]. Rows 0..n_ctx-1
    (the state token and the context tokens) see the prefix and each other; action rows see all."""
    vis = np.ones((suffix_len, prefix_len + suffix_len), dtype=bool)
    vis[:n_ctx, prefix_len + n_ctx:] = False
    return vis


def attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, visible: np.ndarray) -> np.ndarray:
    """R7: q [S][H][D] against the single KV head K, V [P+S][D]; returns o [S][H][D].

    App. A: queries come from the action-noise tokens, keys/values are the LLM layer's KV
    cache concatenated with the suffix tokens' own keys/values.
    """
    S, H, D = q.shape
    scores = (q.reshape(S * H, D) @ K.T).reshape(S, H, -1) / np.sqrt(F64(D))
    scores = np.where(visible[:, None, :], scores, -np.inf)
    scores = scores - scores.max(axis=-1, keepdims=True)
    p = np.exp(scores)
    p = p / p.sum(axis=-1, keepdims=True)
    return (p.reshape(S * H, -1) @ V).reshape(S, H, D)


def gelu_tanh(y: np.ndarray) -> np.ndarray:
    """R8: 0.5 y (1 + tanh(sqrt(2/pi) (y + 0.044715 y^3)))."""
    return 0.5 * y * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (y + 0.044715 * y ** 3)))


def layer_mods(c: np.ndarray, w: dict, layer: int, W: int):
    """R5: the six modulation vectors of one layer for conditioning c."""
    ma = w["attn_mod_w"][layer] @ c + w["attn_mod_b"][layer]
    mm = w["mlp_mod_w"][layer] @ c + w["mlp_mod_b"][layer]
    return ma[:W], ma[W:2 * W], ma[2 * W:], mm[:W], mm[W:2 * W], mm[2 * W:]


def expert_forward(x: np.ndarray, s: np.ndarray, t: float, prefix_k: np.ndarray,
                   prefix_v: np.ndarray, w: dict, cfg, return_hidden: bool = False,
                   corr: np.ndarray | None = None):
    """Velocity v [C][A] of one request at flow time t (App. A, one DiT pass).

    x [C][A] noisy actions, s [S_d] state, prefix_k / prefix_v [L][P][D] the per-layer LLM KV,
    corr [T'][W] the correction items (R15; None or T' = 0: none).
    With return_hidden, also returns the residual stream h [S][W] after the last layer.
    """
    W, H, D = cfg.width, cfg.n_heads, cfg.head_dim
    L, P, C = cfg.n_layers, prefix_k.shape[1], x.shape[0]
    T = 0 if corr is None else corr.shape[0]
    n_ctx = 1 + T
    S = C + n_ctx
    c = time_conditioning(t, w, cfg)
    # R4, R15: row 0 is the state token, rows 1..T' the correction items, then the C action tokens.
    h = np.empty((S, W), dtype=F64)
    h[0] = w["state_in_w"] @ s + w["state_in_b"]
    if T:
        h[1:n_ctx] = corr
    h[n_ctx:] = x @ w["action_in_w"].T + w["action_in_b"]
    visible = suffix_mask(P, S, n_ctx)
    pos = P + np.arange(S)
    for l in range(L):
        sa, ba, ga, sm, bm, gm = layer_mods(c, w, l, W)
        u = rms_modulate(h, sa, ba, cfg.rms_eps)
        q = (u @ w["wq"][l].T).reshape(S, H, D)
        k = u @ w["wk"][l].T
        v = u @ w["wv"][l].T
        q = rope(q, pos, cfg.rope_base)
        k = rope(k, pos, cfg.rope_base)
        K = np.concatenate([prefix_k[l], k], axis=0)
        V = np.concatenate([prefix_v[l], v], axis=0)
        o = attention(q, K, V, visible).reshape(S, H * D)
        h = h + ga * (o @ w["wo"][l].T)
        u = rms_modulate(h, sm, bm, cfg.rms_eps)
        z = gelu_tanh(u @ w["w_gate"][l].T) * (u @ w["w_up"][l].T)
        h = h + gm * (z @ w["w_down"][l].T)
    fm = w["final_mod_w"] @ c + w["final_mod_b"]
    u = rms_modulate(h, fm[:W], fm[W:], cfg.rms_eps)
    vel = u[n_ctx:] @ w["action_out_w"].T + w["action_out_b"]      # R9
    return (vel, h) if return_hidden else vel


def flow_times(num_steps: int) -> np.ndarray:
    """R1: t_k = k / N for k = 0..N-1."""
    return np.arange(num_steps, dtype=F64) / num_steps


def denoise(noise: np.ndarray, s: np.ndarray, num_steps: int, prefix_k: np.ndarray,
            prefix_v: np.ndarray, w: dict, cfg, corr: np.ndarray | None = None) -> np.ndarray:
    """Flow-matching denoise of one request: N Euler steps x <- x + delta v (R1, App. A)."""
    delta = 1.0 / num_steps
    x = noise.astype(F64)
    for t in flow_times(num_steps):
        x = x + delta * expert_forward(x, s, t, prefix_k, prefix_v, w, cfg, corr=corr)
    return x


def to_f64(w: dict) -> dict:
    """Weights as fp64 (per-layer lists preserved); converts tensors on a few threads."""
    from concurrent.futures import ThreadPoolExecutor
    if w.get("__f64__"):
        return w
    with ThreadPoolExecutor(max_workers=8) as ex:
        out = {k: (list(ex.map(lambda a: np.asarray(a, F64), v)) if isinstance(v, list)
                   else np.asarray(v, F64)) for k, v in w.items()}
    out["__f64__"] = True
    return out


def denoise_batch(noise: np.ndarray, state: np.ndarray, num_steps: int, prefix_k: np.ndarray,
                  prefix_v: np.ndarray, w: dict, cfg, corr: np.ndarray | None = None) -> np.ndarray:
    """R10: each request b runs independently. prefix_k/v [L][B][P][D], corr [B][T'][W] or
    None -> actions [B][C][A]."""
    w64 = to_f64(w)
    return np.stack([
        denoise(noise[b], state[b].astype(F64), num_steps,
                prefix_k[:, b].astype(F64), prefix_v[:, b].astype(F64), w64, cfg,
                corr=None if corr is None else corr[b].astype(F64))
        for b in range(noise.shape[0])
    ])


def forward_batch(x: np.ndarray, state: np.ndarray, t: float, prefix_k: np.ndarray,
                  prefix_v: np.ndarray, w: dict, cfg, corr: np.ndarray | None = None):
    """One expert pass per request: returns (v [B][C][A], h [B][S][W])."""
    w64 = to_f64(w)
    vs, hs = [], []
    for b in range(x.shape[0]):
        v, h = expert_forward(x[b].astype(F64), state[b].astype(F64), t,
                              prefix_k[:, b].astype(F64), prefix_v[:, b].astype(F64), w64, cfg,
                              return_hidden=True, corr=None if corr is None else corr[b].astype(F64))
        vs.append(v)
        hs.append(h)
    return np.stack(vs), np.stack(hs)
