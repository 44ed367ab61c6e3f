"""Pins of the CPU oracle against facts fixed outside the oracle itself.

Each test checks the oracle against a closed form, an invariant, a special case that reduces
to a textbook routine, or brute force on tiny inputs, chosen so that a dropped term, a wrong
sign or index, or a transposed operand in the oracle fails at least one of them.
"""

import math
import os

import numpy as np
import pytest
from scipy.special import expit, ndtr

import oracle
from synth import ExpertConfig, PI05, make_requests, make_weights

# Micro expert with every dimension distinct, so a transposed operand cannot pass silently.
MICRO = ExpertConfig(n_layers=2, width=24, n_heads=2, head_dim=8, mlp_dim=40, action_dim=3,
                     state_dim=5, time_dim=12, precision="fp32")


def micro_setup(seed=5, P=6, C=4, B=1, cfg=MICRO, **wkw):
    w = make_weights(cfg, seed, **wkw)
    r = make_requests(cfg, seed + 1, B, P, C)
    return oracle.to_f64(w), r


# ---------------------------------------------------------------- time embedding (R2)

def test_sinusoid_at_t0_is_zero_sines_unit_cosines():
    e = oracle.sinusoidal_time_embedding(0.0, 64, 4e-3, 4.0)
    assert np.all(e[:32] == 0.0) and np.all(e[32:] == 1.0)


def test_sinusoid_points_on_unit_circle():
    for t in (0.13, 0.5, 0.9):
        e = oracle.sinusoidal_time_embedding(t, 64, 4e-3, 4.0)
        np.testing.assert_allclose(e[:32] ** 2 + e[32:] ** 2, 1.0, atol=1e-14)


def test_sinusoid_frequencies_are_geometric_between_the_periods():
    # sin(theta) ~ theta for tiny t, so sin_i / t reads off the angular frequency 2 pi / p_i.
    t, half = 1e-9, 32
    e = oracle.sinusoidal_time_embedding(t, 2 * half, 4e-3, 4.0)
    freq = e[:half] / t
    np.testing.assert_allclose(freq[0], 2 * math.pi / 4e-3, rtol=1e-9)
    np.testing.assert_allclose(freq[-1], 2 * math.pi / 4.0, rtol=1e-9)
    ratio = freq[1:] / freq[:-1]
    np.testing.assert_allclose(ratio, (4e-3 / 4.0) ** (1.0 / (half - 1)), rtol=1e-9)


def test_sinusoid_quarter_periods():
    e = oracle.sinusoidal_time_embedding(1.0, 64, 4e-3, 4.0)       # t = max_period / 4
    assert abs(e[31] - 1.0) < 1e-12 and abs(e[63]) < 1e-12
    e = oracle.sinusoidal_time_embedding(1e-3, 64, 4e-3, 4.0)      # t = min_period / 4
    assert abs(e[0] - 1.0) < 1e-12 and abs(e[32]) < 1e-12


# ---------------------------------------------------------------- time MLP (R3)

def test_time_mlp_single_entry_closed_form_detects_transpose():
    cfg = MICRO
    W = cfg.width
    w = oracle.to_f64(make_weights(cfg, 1))
    z, a, i, j = 0.7, 1.9, 3, 17
    w["time_mlp_in_w"] = np.zeros_like(w["time_mlp_in_w"])
    w["time_mlp_in_b"] = np.full(W, z)
    w["time_mlp_out_w"] = np.zeros((W, W))
    w["time_mlp_out_w"][i, j] = a
    w["time_mlp_out_b"] = np.zeros(W)
    c = oracle.time_conditioning(0.3, w, cfg)
    sw = lambda x: x * expit(x)                       # noqa: E731  swish = x * sigmoid(x)
    expected = np.zeros(W)
    expected[i] = sw(a * sw(z))
    np.testing.assert_allclose(c, expected, atol=1e-15)


# ---------------------------------------------------------------- GeGLU (R8)

def test_gelu_tanh_against_exact_gelu_bound():
    y = np.linspace(-8, 8, 4001)
    exact = y * ndtr(y)                               # x * Phi(x), the erf form of GELU
    err = np.abs(oracle.gelu_tanh(y) - exact)
    # The tanh approximation stays within about 3e-4 of the exact GELU on the real line.
    assert err.max() < 5e-4
    assert err.max() > 1e-5                           # it is the approximation, not erf
    assert oracle.gelu_tanh(np.array([0.0]))[0] == 0.0


# ---------------------------------------------------------------- adaptive RMSNorm (R5)

def test_rms_modulate_unit_rms_with_zero_modulation():
    rng = np.random.default_rng(0)
    h = rng.standard_normal((5, 24)) * 3.0
    u = oracle.rms_modulate(h, np.zeros(24), np.zeros(24), 0.0)
    np.testing.assert_allclose(np.mean(u * u, axis=-1), 1.0, rtol=1e-13)


def test_rms_modulate_scale_invariant_and_closed_form_on_constant_rows():
    rng = np.random.default_rng(1)
    h = rng.standard_normal((3, 24))
    sig, bet = rng.standard_normal(24), rng.standard_normal(24)
    np.testing.assert_allclose(oracle.rms_modulate(7.5 * h, sig, bet, 0.0),
                               oracle.rms_modulate(h, sig, bet, 0.0), rtol=1e-12)
    # A constant row c normalises to sign(c) / sqrt(1 + eps / c^2): u = that * (1 + sigma) + beta.
    eps, c = 1e-2, -0.3
    u = oracle.rms_modulate(np.full((1, 24), c), sig, bet, eps)
    r = c / math.sqrt(c * c + eps)
    np.testing.assert_allclose(u[0], r * (1 + sig) + bet, rtol=1e-13)


# ---------------------------------------------------------------- rotary encoding (R6)

def test_rope_closed_form_d4():
    # D = 4, base 100: pair (x0, x2) turns by pos * 1, pair (x1, x3) by pos * 100^(-1/2).
    x = np.array([[1.0, 2.0, 3.0, 4.0]])
    pos = 3
    out = oracle.rope(x, np.array([pos]), 100.0)[0]
    a0, a1 = pos * 1.0, pos * 0.1
    exp = [1 * math.cos(a0) - 3 * math.sin(a0), 2 * math.cos(a1) - 4 * math.sin(a1),
           3 * math.cos(a0) + 1 * math.sin(a0), 4 * math.cos(a1) + 2 * math.sin(a1)]
    np.testing.assert_allclose(out, exp, rtol=1e-14)


def test_rope_identity_at_zero_norm_preserving_and_relative():
    rng = np.random.default_rng(2)
    q, k = rng.standard_normal((1, 16)), rng.standard_normal((1, 16))
    np.testing.assert_array_equal(oracle.rope(q, np.array([0]), 1e4), q)
    r = oracle.rope(q, np.array([37]), 1e4)
    np.testing.assert_allclose(np.linalg.norm(r), np.linalg.norm(q), rtol=1e-14)
    d1 = oracle.rope(q, np.array([9]), 1e4) @ oracle.rope(k, np.array([4]), 1e4).T
    d2 = oracle.rope(q, np.array([109]), 1e4) @ oracle.rope(k, np.array([104]), 1e4).T
    np.testing.assert_allclose(d1, d2, rtol=1e-11)
    np.testing.assert_array_equal(oracle.rope(q, np.array([5]), 0.0), q)


# ---------------------------------------------------------------- attention (R7)

def brute_force_attention(q, K, V, P):
    """Scalar loops: softmax over the visible keys of each (row, head)."""
    S, H, D = q.shape
    o = np.zeros_like(q)
    for i in range(S):
        n_vis = P + 1 if i == 0 else K.shape[0]
        for hh in range(H):
            sc = [sum(q[i, hh, d] * K[n, d] for d in range(D)) / math.sqrt(D) for n in range(n_vis)]
            m = max(sc)
            ex = [math.exp(s - m) for s in sc]
            tot = sum(ex)
            for d in range(D):
                o[i, hh, d] = sum(ex[n] * V[n, d] for n in range(n_vis)) / tot
    return o


def test_attention_matches_brute_force_with_state_row_mask():
    rng = np.random.default_rng(3)
    P, S, H, D = 5, 4, 2, 8
    q = rng.standard_normal((S, H, D)) * 2
    K, V = rng.standard_normal((P + S, D)), rng.standard_normal((P + S, D))
    o = oracle.attention(q, K, V, oracle.suffix_mask(P, S))
    np.testing.assert_allclose(o, brute_force_attention(q, K, V, P), rtol=1e-12, atol=1e-13)


def test_attention_zero_query_averages_visible_values():
    rng = np.random.default_rng(4)
    P, S, H, D = 6, 3, 2, 8
    K, V = rng.standard_normal((P + S, D)), rng.standard_normal((P + S, D))
    o = oracle.attention(np.zeros((S, H, D)), K, V, oracle.suffix_mask(P, S))
    np.testing.assert_allclose(o[0, 0], V[:P + 1].mean(0), rtol=1e-13)
    np.testing.assert_allclose(o[2, 1], V.mean(0), rtol=1e-13)


def test_attention_two_key_closed_form_fixes_the_scale():
    # Prefix of 1 key; row 0 sees key 0 and itself: o = V0 + (V1 - V0) * sigmoid((s1 - s0)/sqrt(D)).
    D = 16
    q = np.zeros((1, 1, D))
    q[0, 0, 0] = 3.0
    K = np.zeros((2, D))
    K[0, 0], K[1, 0] = 0.5, 2.0
    V = np.arange(2 * D, dtype=float).reshape(2, D)
    o = oracle.attention(q, K, V, oracle.suffix_mask(1, 1))
    g = expit((3.0 * 2.0 - 3.0 * 0.5) / math.sqrt(D))
    np.testing.assert_allclose(o[0, 0], V[0] + (V[1] - V[0]) * g, rtol=1e-13)


def test_attention_prefix_permutation_invariance():
    rng = np.random.default_rng(6)
    P, S, H, D = 7, 3, 2, 8
    q = rng.standard_normal((S, H, D))
    K, V = rng.standard_normal((P + S, D)), rng.standard_normal((P + S, D))
    perm = np.concatenate([rng.permutation(P), np.arange(P, P + S)])
    m = oracle.suffix_mask(P, S)
    np.testing.assert_allclose(oracle.attention(q, K[perm], V[perm], m),
                               oracle.attention(q, K, V, m), rtol=1e-12)


# ---------------------------------------------------------------- whole expert / integrator

@pytest.mark.parametrize("N", [1, 3, 10])
def test_zero_velocity_head_gives_closed_form_integral(N):
    # W_out = 0, b_out = c  =>  v = c at every step  =>  x_N = x_0 + N * (1/N) * c = x_0 + c.
    w, r = micro_setup()
    c = np.array([0.25, -1.5, 3.0])
    w["action_out_w"] = np.zeros_like(w["action_out_w"])
    w["action_out_b"] = c
    x = oracle.denoise(r["noise"][0].astype(float), r["state"][0].astype(float), N,
                       r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    np.testing.assert_allclose(x, r["noise"][0] + c, rtol=1e-13, atol=1e-14)


def test_one_step_equals_one_forward_at_t0():
    w, r = micro_setup()
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x0, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    x1 = oracle.denoise(x0, s, 1, *args)
    np.testing.assert_allclose(x1, x0 + oracle.expert_forward(x0, s, 0.0, *args), rtol=1e-14)


def test_later_steps_use_later_times():
    # With two steps, the second velocity is taken at t = 1/2 on x_1.
    w, r = micro_setup()
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x0, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    x1 = x0 + 0.5 * oracle.expert_forward(x0, s, 0.0, *args)
    x2 = x1 + 0.5 * oracle.expert_forward(x1, s, 0.5, *args)
    np.testing.assert_allclose(oracle.denoise(x0, s, 2, *args), x2, rtol=1e-14)


def test_zero_gates_make_every_layer_the_identity():
    # gamma = 0 for both sublayers (zero gate rows and zero gate biases) => h stays the embedding.
    w, r = micro_setup()
    W = MICRO.width
    for l in range(MICRO.n_layers):
        for mw, mb in (("attn_mod_w", "attn_mod_b"), ("mlp_mod_w", "mlp_mod_b")):
            w[mw][l][2 * W:] = 0.0
            w[mb][l][2 * W:] = 0.0
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    _, h = oracle.expert_forward(x, s, 0.4, r["prefix_k"][:, 0].astype(float),
                                 r["prefix_v"][:, 0].astype(float), w, MICRO, return_hidden=True)
    np.testing.assert_allclose(h[0], w["state_in_w"] @ s + w["state_in_b"], rtol=1e-14)
    np.testing.assert_allclose(h[1:], x @ w["action_in_w"].T + w["action_in_b"], rtol=1e-14)


def test_velocity_through_identity_layers_by_scalar_loops():
    # With both gates zero every layer is the identity, so the velocity of action j is the final
    # norm of its embedding: u = e / rms(e) * (1 + sigma_f) + beta_f with (sigma_f, beta_f) the
    # first and second halves of M_f c + m_f (R5), then v = W_out u + b_out. Rebuilt by loops.
    w, r = micro_setup(mod_bias_std=0.7)
    W, A = MICRO.width, MICRO.action_dim
    for l in range(MICRO.n_layers):
        for mw, mb in (("attn_mod_w", "attn_mod_b"), ("mlp_mod_w", "mlp_mod_b")):
            w[mw][l][2 * W:] = 0.0
            w[mb][l][2 * W:] = 0.0
    t = 0.3
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    v = oracle.expert_forward(x, s, t, r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float),
                              w, MICRO)
    c = oracle.time_conditioning(t, w, MICRO)
    fm = [sum(w["final_mod_w"][i][k] * c[k] for k in range(W)) + w["final_mod_b"][i] for i in range(2 * W)]
    for j in range(x.shape[0]):
        e = [sum(w["action_in_w"][i][a] * x[j][a] for a in range(A)) + w["action_in_b"][i] for i in range(W)]
        rms = math.sqrt(sum(q * q for q in e) / W + MICRO.rms_eps)
        u = [e[i] / rms * (1.0 + fm[i]) + fm[W + i] for i in range(W)]
        want = [sum(w["action_out_w"][a][i] * u[i] for i in range(W)) + w["action_out_b"][a] for a in range(A)]
        np.testing.assert_allclose(v[j], want, rtol=1e-12, atol=1e-13)


def test_state_row_does_not_see_the_actions():
    w, r = micro_setup(mod_bias_std=1.0)
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    _, h1 = oracle.expert_forward(x, s, 0.2, *args, return_hidden=True)
    _, h2 = oracle.expert_forward(x + 1.0, s, 0.2, *args, return_hidden=True)
    np.testing.assert_array_equal(h1[0], h2[0])
    assert np.abs(h1[1:] - h2[1:]).max() > 1e-3
    _, h3 = oracle.expert_forward(x, s + 1.0, 0.2, *args, return_hidden=True)
    assert np.abs(h1[1:] - h3[1:]).max() > 1e-6          # the actions do see the state


def test_prefix_kv_of_every_layer_is_used():
    w, r = micro_setup(mod_bias_std=1.0)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    K, V = r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float)
    v0 = oracle.expert_forward(x, s, 0.1, K, V, w, MICRO)
    for l in range(MICRO.n_layers):
        V2 = V.copy()
        V2[l] += 1.0
        assert np.abs(oracle.expert_forward(x, s, 0.1, K, V2, w, MICRO) - v0).max() > 1e-6


def test_batch_requests_are_independent():
    cfg = MICRO
    w = make_weights(cfg, 9)
    rb = make_requests(cfg, 10, 3, 6, 4)
    out = oracle.denoise_batch(rb["noise"], rb["state"], 3, rb["prefix_k"], rb["prefix_v"], w, cfg)
    r1 = make_requests(cfg, 10, 1, 6, 4, first_request=2)
    one = oracle.denoise_batch(r1["noise"], r1["state"], 3, r1["prefix_k"], r1["prefix_v"], w, cfg)
    np.testing.assert_array_equal(out[2], one[0])


def test_time_enters_only_through_the_conditioning():
    # All time-MLP weights and biases zero => c = swish(0) = 0 => v does not depend on t.
    w, r = micro_setup()
    for k in ("time_mlp_in_w", "time_mlp_in_b", "time_mlp_out_w", "time_mlp_out_b"):
        w[k] = np.zeros_like(w[k])
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    np.testing.assert_array_equal(oracle.expert_forward(x, s, 0.0, *args),
                                  oracle.expert_forward(x, s, 0.7, *args))


# ---------------------------------------------------------------- the paper's dimensions

def test_pi05_dimensions_match_the_paper_table():
    path = os.path.join(os.path.dirname(__file__), "golden", "pi05_action_expert_dims.txt")
    vals = {}
    for line in open(path):
        line = line.split("#")[0].strip()
        if line:
            k, v = line.split("=")
            vals[k.strip()] = int(v)
    assert PI05.n_layers == vals["layers"]
    assert PI05.width == vals["width"]
    assert PI05.n_heads == vals["heads"]
    assert PI05.head_dim == vals["head_dim"]
    assert vals["denoise_steps"] == 10


def test_one_layer_wiring_from_pinned_parts():
    # One layer, rebuilt from parts pinned above (RMS modulation, rotary encoding, brute-force
    # attention, tanh GELU) with the split order (sigma, beta, gamma), positions P + i,
    # keys [prefix ; suffix] and both gates spelled out here.
    cfg = MICRO.with_(n_layers=1)
    P, C = 4, 3
    w = oracle.to_f64(make_weights(cfg, 21, mod_bias_std=1.0))
    r = make_requests(cfg, 22, 1, P, C)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    K0, V0 = r["prefix_k"][0, 0].astype(float), r["prefix_v"][0, 0].astype(float)
    W, H, D, S = cfg.width, cfg.n_heads, cfg.head_dim, C + 1
    c = oracle.time_conditioning(0.6, w, cfg)
    h = np.vstack([w["state_in_w"] @ s + w["state_in_b"], x @ w["action_in_w"].T + w["action_in_b"]])
    ma = w["attn_mod_w"][0] @ c + w["attn_mod_b"][0]
    mm = w["mlp_mod_w"][0] @ c + w["mlp_mod_b"][0]
    u = oracle.rms_modulate(h, ma[:W], ma[W:2 * W], cfg.rms_eps)
    pos = np.arange(P, P + S)
    q = oracle.rope((u @ w["wq"][0].T).reshape(S, H, D), pos, cfg.rope_base)
    k = oracle.rope(u @ w["wk"][0].T, pos, cfg.rope_base)
    v = u @ w["wv"][0].T
    o = brute_force_attention(q, np.vstack([K0, k]), np.vstack([V0, v]), P)
    h = h + ma[2 * W:] * (o.reshape(S, H * D) @ w["wo"][0].T)
    u = oracle.rms_modulate(h, mm[:W], mm[W:2 * W], cfg.rms_eps)
    g, up = u @ w["w_gate"][0].T, u @ w["w_up"][0].T
    h = h + mm[2 * W:] * ((oracle.gelu_tanh(g) * up) @ w["w_down"][0].T)
    _, h_or = oracle.expert_forward(x, s, 0.6, r["prefix_k"][:, 0].astype(float),
                                    r["prefix_v"][:, 0].astype(float), w, cfg, return_hidden=True)
    np.testing.assert_allclose(h_or, h, rtol=1e-11, atol=1e-12)


def test_velocity_of_action_j_comes_from_token_j():
    # With both gates zero every layer is the identity, so v_j depends on x_j alone.
    w, r = micro_setup()
    W = MICRO.width
    for l in range(MICRO.n_layers):
        for mw, mb in (("attn_mod_w", "attn_mod_b"), ("mlp_mod_w", "mlp_mod_b")):
            w[mw][l][2 * W:] = 0.0
            w[mb][l][2 * W:] = 0.0
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    v0 = oracle.expert_forward(x, s, 0.3, *args)
    for j in range(x.shape[0]):
        x2 = x.copy()
        x2[j] += 0.5
        d = np.abs(oracle.expert_forward(x2, s, 0.3, *args) - v0).max(axis=1)
        assert d[j] > 1e-6 and np.all(np.delete(d, j) == 0.0)


# ---------------------------------------------------------------- correction items (R15)

def _corr(T, W, seed=31):
    return np.random.default_rng(seed).normal(0.0, 1.0, (T, W))


def _identity_layers(w, cfg):
    """Both sublayer gates zero: every layer is the identity on the residual stream."""
    W = cfg.width
    for l in range(cfg.n_layers):
        for mw, mb in (("attn_mod_w", "attn_mod_b"), ("mlp_mod_w", "mlp_mod_b")):
            w[mw][l][2 * W:] = 0.0
            w[mb][l][2 * W:] = 0.0
    return w


def test_no_correction_items_is_the_plain_expert():
    w, r = micro_setup(mod_bias_std=1.0)
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    v0, h0 = oracle.expert_forward(x, s, 0.4, *args, return_hidden=True)
    v1, h1 = oracle.expert_forward(x, s, 0.4, *args, return_hidden=True,
                                   corr=np.zeros((0, MICRO.width)))
    np.testing.assert_array_equal(v0, v1)
    np.testing.assert_array_equal(h0, h1)


def test_correction_items_enter_the_residual_stream_unchanged():
    # With identity layers the stream after the last layer is its input: state embedding,
    # the items as given, the action embeddings; the velocity is the plain expert's.
    w, r = micro_setup()
    w = _identity_layers(w, MICRO)
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    corr = _corr(3, MICRO.width)
    v, h = oracle.expert_forward(x, s, 0.3, *args, return_hidden=True, corr=corr)
    assert h.shape == (1 + 3 + x.shape[0], MICRO.width)
    np.testing.assert_allclose(h[0], w["state_in_w"] @ s + w["state_in_b"], rtol=1e-14)
    np.testing.assert_array_equal(h[1:4], corr)
    np.testing.assert_allclose(h[4:], x @ w["action_in_w"].T + w["action_in_b"], rtol=1e-14)
    np.testing.assert_allclose(v, oracle.expert_forward(x, s, 0.3, *args), rtol=1e-14)


def test_context_rows_do_not_see_the_actions_and_the_actions_see_every_item():
    w, r = micro_setup(mod_bias_std=1.0)
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, MICRO)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    corr = _corr(3, MICRO.width)
    v1, h1 = oracle.expert_forward(x, s, 0.2, *args, return_hidden=True, corr=corr)
    v2, h2 = oracle.expert_forward(x + 1.0, s, 0.2, *args, return_hidden=True, corr=corr)
    np.testing.assert_array_equal(h1[:4], h2[:4])          # state and context rows
    assert np.abs(h1[4:] - h2[4:]).max() > 1e-3
    for j in range(3):
        c2 = corr.copy()
        c2[j] += 0.5
        v3, h3 = oracle.expert_forward(x, s, 0.2, *args, return_hidden=True, corr=c2)
        assert np.abs(v3 - v1).max() > 1e-6                # every item reaches the actions
        assert np.abs(h3[0] - h1[0]).max() > 1e-6          # and the state row sees it


def test_correction_items_are_an_unordered_set_without_rope():
    # Without position encoding attention does not depend on key order, so permuting the
    # items permutes their rows of the stream and leaves the velocity unchanged.
    cfg = MICRO.with_(rope_base=0.0)
    w, r = micro_setup(cfg=cfg, mod_bias_std=1.0)
    args = (r["prefix_k"][:, 0].astype(float), r["prefix_v"][:, 0].astype(float), w, cfg)
    x, s = r["noise"][0].astype(float), r["state"][0].astype(float)
    corr = _corr(4, cfg.width)
    perm = np.array([2, 0, 3, 1])
    v1, h1 = oracle.expert_forward(x, s, 0.5, *args, return_hidden=True, corr=corr)
    v2, h2 = oracle.expert_forward(x, s, 0.5, *args, return_hidden=True, corr=corr[perm])
    np.testing.assert_allclose(v2, v1, rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(h2[1:5], h1[1:5][perm], rtol=1e-11, atol=1e-13)
