"""Pins of the LLM-prefill oracle (oracle/prefill.py) against facts fixed outside it: a
brute-force scalar rebuild of a layer on tiny inputs, the closed form when every layer is the
identity, permutation equivariance of the bidirectional prefix without rotary coding, the
reach of the last token to the first, and the paper's printed dimensions."""

import math
import os

import numpy as np

import oracle.prefill as pf
from synth import GEMMA2B, llm_weight_shapes, make_llm_weights, make_prefix_embeddings

MICRO = GEMMA2B.with_(n_layers=2, width=6, n_heads=2, head_dim=4, mlp_dim=5, precision="fp32")


def setup(cfg=MICRO, seed=3, P=4, norm_std=0.3):
    w = pf.to_f64_llm(make_llm_weights(cfg, seed, std=0.4, norm_std=norm_std))
    x = make_prefix_embeddings(cfg, seed + 1, 1, P)[0].astype(np.float64)
    return w, x


# ---------------------------------------------------------------- scalar brute force

def bf_rms(row, scale, eps):
    r = math.sqrt(sum(v * v for v in row) / len(row) + eps)
    return [v / r * (1.0 + s) for v, s in zip(row, scale)]


def bf_matvec(Wm, v):
    return [sum(Wm[i][j] * v[j] for j in range(len(v))) for i in range(len(Wm))]


def bf_rope(vec, p, base):
    D = len(vec)
    half = D // 2
    out = list(vec)
    for d in range(half):
        ang = p * base ** (-2.0 * d / D)
        a, b = vec[d], vec[d + half]
        out[d] = a * math.cos(ang) - b * math.sin(ang)
        out[d + half] = b * math.cos(ang) + a * math.sin(ang)
    return out


def bf_gelu(y):
    return 0.5 * y * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) * (y + 0.044715 * y ** 3)))


def bf_layer(h, w, l, cfg):
    """One Gemma block on token rows h (lists), by loops: returns (K rows, V rows, new h)."""
    P, H, D = len(h), cfg.n_heads, cfg.head_dim
    u = [bf_rms(h[p], w["attn_norm"][l], cfg.rms_eps) for p in range(P)]
    q = [bf_matvec(w["wq"][l], u[p]) for p in range(P)]
    k = [bf_rope(bf_matvec(w["wk"][l], u[p]), p, cfg.rope_base) for p in range(P)]
    v = [bf_matvec(w["wv"][l], u[p]) for p in range(P)]
    o = []
    for p in range(P):
        row = []
        for hd in range(H):
            qh = bf_rope(q[p][hd * D:(hd + 1) * D], p, cfg.rope_base)
            s = [sum(qh[d] * k[n][d] for d in range(D)) / math.sqrt(D) for n in range(P)]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            row += [sum(e[n] / z * v[n][d] for n in range(P)) for d in range(D)]
        o.append(row)
    h1 = [[a + b for a, b in zip(h[p], bf_matvec(w["wo"][l], o[p]))] for p in range(P)]
    u2 = [bf_rms(h1[p], w["mlp_norm"][l], cfg.rms_eps) for p in range(P)]
    z = [[bf_gelu(g) * up for g, up in zip(bf_matvec(w["w_gate"][l], u2[p]), bf_matvec(w["w_up"][l], u2[p]))]
         for p in range(P)]
    h2 = [[a + b for a, b in zip(h1[p], bf_matvec(w["w_down"][l], z[p]))] for p in range(P)]
    return k, v, h2


def test_two_layers_by_scalar_brute_force():
    w, x = setup()
    K, V, out = pf.llm_prefill(x, w, MICRO, return_output=True)
    h = [list(r) for r in x]
    for l in range(MICRO.n_layers):
        k, v, h = bf_layer(h, w, l, MICRO)
        np.testing.assert_allclose(K[l], np.array(k), rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(V[l], np.array(v), rtol=1e-11, atol=1e-13)
    want = [bf_rms(r, w["final_norm"], MICRO.rms_eps) for r in h]
    np.testing.assert_allclose(out, np.array(want), rtol=1e-11, atol=1e-13)


def test_identity_layers_cache_the_normalised_input():
    # Zero output and down projections: every layer passes the stream through, so layer l
    # caches rope(rms(x)(1 + a_l) Wk_l) and rms(x)(1 + a_l) Wv_l.
    w, x = setup()
    for l in range(MICRO.n_layers):
        w["wo"][l] = np.zeros_like(w["wo"][l])
        w["w_down"][l] = np.zeros_like(w["w_down"][l])
    K, V, out = pf.llm_prefill(x, w, MICRO, return_output=True)
    for l in range(MICRO.n_layers):
        for p in range(x.shape[0]):
            u = bf_rms(list(x[p]), w["attn_norm"][l], MICRO.rms_eps)
            np.testing.assert_allclose(K[l, p], bf_rope(bf_matvec(w["wk"][l], u), p, MICRO.rope_base),
                                       rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(V[l, p], bf_matvec(w["wv"][l], u), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(out[0], bf_rms(list(x[0]), w["final_norm"], MICRO.rms_eps), rtol=1e-12)


def test_bidirectional_prefix_is_permutation_equivariant_without_rope():
    cfg = MICRO.with_(rope_base=0.0)
    w, x = setup(cfg=cfg, P=5)
    perm = np.array([3, 0, 4, 2, 1])
    K1, V1, o1 = pf.llm_prefill(x, w, cfg, return_output=True)
    K2, V2, o2 = pf.llm_prefill(x[perm], w, cfg, return_output=True)
    np.testing.assert_allclose(K2, K1[:, perm], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(V2, V1[:, perm], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(o2, o1[perm], rtol=1e-11, atol=1e-13)


def test_the_first_token_sees_the_last():
    w, x = setup(P=5)
    K1, _ = pf.llm_prefill(x, w, MICRO)
    x2 = x.copy()
    x2[-1] += 1.0
    K2, _ = pf.llm_prefill(x2, w, MICRO)
    np.testing.assert_array_equal(K1[0, 0], K2[0, 0])    # layer 0 caches token 0's own input
    assert np.abs(K1[1, 0] - K2[1, 0]).max() > 1e-6      # layer 1 has seen the last token


def test_batch_requests_are_independent():
    cfg = MICRO
    w = make_llm_weights(cfg, 7, std=0.4, norm_std=0.3)
    x = make_prefix_embeddings(cfg, 8, 3, 4)
    K, V, out = pf.prefill_batch(x, w, cfg)
    K1, V1, out1 = pf.prefill_batch(x[2:3], w, cfg)
    np.testing.assert_array_equal(K[:, 2], K1[:, 0])
    np.testing.assert_array_equal(out[2], out1[0])


def test_gemma2b_dimensions_match_the_paper_table():
    path = os.path.join(os.path.dirname(__file__), "golden", "pi05_llm_dims.txt")
    dims = {}
    for line in open(path):
        line = line.split("#")[0].strip()
        if line:
            k, v = (s.strip() for s in line.split("="))
            dims[k] = int(v)
    assert (GEMMA2B.n_layers, GEMMA2B.width, GEMMA2B.n_heads, GEMMA2B.head_dim) == (
        dims["layers"], dims["width"], dims["heads"], dims["head_dim"])
    shapes = llm_weight_shapes(GEMMA2B)
    layer_params = GEMMA2B.n_layers * sum(int(np.prod(s)) for k, s in shapes.items() if k != "final_norm")
    assert 1.9e9 < layer_params < 2.1e9          # "Gemma 2B" (token embeddings are inputs here)
