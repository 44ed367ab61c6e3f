"""Pins of the future-correction oracle (oracle/correction.py) against facts fixed outside it:
scalar brute-force rebuilds of the compressor and of the module on tiny inputs, invariances
that softmax attention and LayerNorm guarantee, which actions reach the last token, the
compressed tokens' symmetry, and the paper's printed sizes."""

import math
import os

import numpy as np
import pytest

import oracle.correction as oc
from synth import GEMMA2B, PI05
from synth.correction import (PI05_CORRECTION, correction_param_count, make_correction_inputs,
                              make_correction_weights)

MICRO = PI05_CORRECTION.with_(width=4, n_heads=2, head_dim=2, mlp_dim=6, d_vlm=5, n_items=2,
                              action_dim=3, max_delta=6, precision="fp32")


def setup(cfg=MICRO, seed=5, T=3, delta=4):
    w = oc.to_f64_corr(make_correction_weights(cfg, seed, std=0.5, bias_std=0.3, norm_std=0.3))
    inp = make_correction_inputs(cfg, seed + 1, 1, T, delta)
    return w, {k: v[0].astype(np.float64) for k, v in inp.items()}


# ---------------------------------------------------------------- scalar brute force

def bf_ln(row, g, b, eps):
    n = len(row)
    mu = sum(row) / n
    var = sum((v - mu) ** 2 for v in row) / n
    return [(v - mu) / math.sqrt(var + eps) * gi + bi for v, gi, bi in zip(row, g, b)]


def bf_affine(Wm, v, bias):
    return [sum(Wm[i][j] * v[j] for j in range(len(v))) + bias[i] for i in range(len(Wm))]


def bf_gelu(y):
    return 0.5 * y * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) * (y + 0.044715 * y ** 3)))


def bf_mha(xq, xkv, w, p, cfg):
    H, Dh = cfg.n_heads, cfg.head_dim
    q = [bf_affine(w[p + "wq"], r, w[p + "bq"]) for r in xq]
    k = [bf_affine(w[p + "wk"], r, w[p + "bk"]) for r in xkv]
    v = [bf_affine(w[p + "wv"], r, w[p + "bv"]) for r in xkv]
    out = []
    for i in range(len(xq)):
        cat = []
        for h in range(H):
            sl = slice(h * Dh, (h + 1) * Dh)
            s = [sum(a * c for a, c in zip(q[i][sl], k[j][sl])) / math.sqrt(Dh) for j in range(len(xkv))]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            cat += [sum(e[j] / z * v[j][sl][d] for j in range(len(xkv))) for d in range(Dh)]
        out.append(bf_affine(w[p + "wo"], cat, w[p + "bo"]))
    return out


def bf_mlp(row, w, p):
    hid = [bf_gelu(y) for y in bf_affine(w[p + "w1"], row, w[p + "b1"])]
    return bf_affine(w[p + "w2"], hid, w[p + "b2"])


def bf_add(a, b):
    return [[x + y for x, y in zip(r, s)] for r, s in zip(a, b)]


def bf_block(x, w, p, cfg):
    u = [bf_ln(r, w[p + "ln1_w"], w[p + "ln1_b"], cfg.ln_eps) for r in x]
    x = bf_add(x, bf_mha(u, u, w, p + "sa_", cfg))
    u = [bf_ln(r, w[p + "ln2_w"], w[p + "ln2_b"], cfg.ln_eps) for r in x]
    return bf_add(x, [bf_mlp(r, w, p + "mlp_") for r in u])


def bf_compress(hv, w, cfg):
    x = [list(r) for r in w["qf_query"]]
    u = [bf_ln(r, w["qf_ln1_w"], w["qf_ln1_b"], cfg.ln_eps) for r in x]
    x = bf_add(x, bf_mha(u, u, w, "qf_sa_", cfg))
    u = [bf_ln(r, w["qf_ln2_w"], w["qf_ln2_b"], cfg.ln_eps) for r in x]
    x = bf_add(x, bf_mha(u, [list(r) for r in hv], w, "qf_ca_", cfg))
    u = [bf_ln(r, w["qf_ln3_w"], w["qf_ln3_b"], cfg.ln_eps) for r in x]
    x = bf_add(x, [bf_mlp(r, w, "qf_mlp_") for r in u])
    return [bf_ln(r, w["qf_lnf_w"], w["qf_lnf_b"], cfg.ln_eps) for r in x]


def bf_correct(hc, acts, w, cfg):
    n = len(acts)
    tok = []
    for k, a in enumerate(acts):
        hid = [bf_gelu(y) for y in bf_affine(w["act_w1"], list(a), w["act_b1"])]
        e = bf_affine(w["act_w2"], hid, w["act_b2"])
        tok.append([x + pe for x, pe in zip(e, w["act_pos"][k])])
    s = bf_block(tok, w, "ab_", cfg)[n - 1]
    x = [bf_affine(w["fuse_w"], list(r) + s, w["fuse_b"]) for r in hc]
    for i in range(cfg.n_joint):
        x = bf_block(x, w, f"jb{i}_", cfg)
    u = [bf_ln(r, w["head_ln_w"], w["head_ln_b"], cfg.ln_eps) for r in x]
    hf = [bf_affine(w["corr_w"], r, w["corr_b"]) for r in u]
    pooled = [sum(r[d] for r in u) / len(u) for d in range(cfg.width)]
    conf = sum(c * p for c, p in zip(w["conf_w"][0], pooled)) + w["conf_b"][0]
    return hf, conf


def test_compressor_by_scalar_brute_force():
    w, inp = setup(T=3)
    got = oc.qformer_compress(inp["h_vlm"], w, MICRO)
    assert got.shape == (MICRO.n_items, MICRO.width)
    np.testing.assert_allclose(got, np.array(bf_compress(inp["h_vlm"], w, MICRO)), rtol=1e-11, atol=1e-13)


@pytest.mark.parametrize("delta", [1, 4, 6])
def test_correction_module_by_scalar_brute_force(delta):
    w, inp = setup(delta=delta)
    hf, conf = oc.future_correction(inp["h_c"], inp["actions"], w, MICRO)
    want_h, want_c = bf_correct(inp["h_c"], inp["actions"], w, MICRO)
    np.testing.assert_allclose(hf, np.array(want_h), rtol=1e-11, atol=1e-13)
    assert conf == pytest.approx(want_c, rel=1e-11, abs=1e-13)


def test_vlm_branch_chains_compressor_and_module():
    w, inp = setup(T=3, delta=2)
    hf, conf = oc.correct_from_vlm(inp["h_vlm"], inp["actions"], w, MICRO)
    want_h, want_c = bf_correct(bf_compress(inp["h_vlm"], w, MICRO), inp["actions"], w, MICRO)
    np.testing.assert_allclose(hf, np.array(want_h), rtol=1e-11, atol=1e-13)
    assert conf == pytest.approx(want_c, rel=1e-11, abs=1e-13)


# ---------------------------------------------------------------- invariances

def test_compressor_ignores_the_order_of_vlm_tokens():
    w, inp = setup(T=5)
    perm = np.array([2, 4, 0, 1, 3])
    a = oc.qformer_compress(inp["h_vlm"], w, MICRO)
    b = oc.qformer_compress(inp["h_vlm"][perm], w, MICRO)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-14)


def test_duplicating_every_vlm_token_changes_nothing():
    # Softmax attention weighs each distinct key by its normalised share: two copies of every
    # token give each copy half the weight.
    w, inp = setup(T=3)
    a = oc.qformer_compress(inp["h_vlm"], w, MICRO)
    b = oc.qformer_compress(np.concatenate([inp["h_vlm"], inp["h_vlm"]]), w, MICRO)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-14)


def test_one_vlm_token_makes_the_cross_attention_query_free():
    # With a single key every query takes all of its value, so the query and key projections of
    # the cross-attention drop out.
    w, inp = setup(T=1)
    a = oc.qformer_compress(inp["h_vlm"], w, MICRO)
    w2 = dict(w)
    w2["qf_ca_wq"] = np.zeros_like(w["qf_ca_wq"])
    w2["qf_ca_wk"] = 3.0 * w["qf_ca_wk"]
    w2["qf_ca_bk"] = -w["qf_ca_bk"]
    b = oc.qformer_compress(inp["h_vlm"], w2, MICRO)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-14)


def test_key_bias_drops_out_of_every_attention():
    # q . (k + b_k) adds q . b_k to every score of a query alike; softmax cancels it.
    w, inp = setup(T=3, delta=3)
    a = oc.correct_from_vlm(inp["h_vlm"], inp["actions"], w, MICRO)
    w2 = dict(w)
    for name in [k for k in w if k.endswith("bk")]:
        w2[name] = w[name] + 7.0
    b = oc.correct_from_vlm(inp["h_vlm"], inp["actions"], w2, MICRO)
    np.testing.assert_allclose(b[0], a[0], rtol=1e-10, atol=1e-12)
    assert b[1] == pytest.approx(a[1], rel=1e-10, abs=1e-12)


def test_layer_norm_is_shift_and_scale_invariant():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((3, 8))
    g, b = rng.standard_normal(8), rng.standard_normal(8)
    a = oc.layer_norm(x, g, b, 0.0)
    np.testing.assert_allclose(oc.layer_norm(2.5 * x - 1.75, g, b, 0.0), a, rtol=1e-12, atol=1e-13)
    z = oc.layer_norm(x, np.ones(8), np.zeros(8), 0.0)
    np.testing.assert_allclose(z.mean(axis=1), 0.0, atol=1e-13)
    np.testing.assert_allclose((z ** 2).mean(axis=1), 1.0, rtol=1e-12)


def test_only_the_position_table_orders_the_earlier_actions():
    # Without position rows, attention treats the actions before the last as a set; with them,
    # their order matters; and every action, first or last, reaches the output.
    w, inp = setup(delta=5)
    acts = inp["actions"]
    perm = np.array([3, 0, 2, 1, 4])
    base = oc.future_correction(inp["h_c"], acts, w, MICRO)[0]
    moved = oc.future_correction(inp["h_c"], acts[perm], w, MICRO)[0]
    assert np.abs(base - moved).max() > 1e-6
    w0 = dict(w)
    w0["act_pos"] = np.zeros_like(w["act_pos"])
    a = oc.future_correction(inp["h_c"], acts, w0, MICRO)[0]
    b = oc.future_correction(inp["h_c"], acts[perm], w0, MICRO)[0]
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-14)
    swap_last = np.array([0, 1, 2, 4, 3])
    c = oc.future_correction(inp["h_c"], acts[swap_last], w0, MICRO)[0]
    assert np.abs(a - c).max() > 1e-6
    first = acts.copy()
    first[0] += 1.0
    d = oc.future_correction(inp["h_c"], first, w, MICRO)[0]
    assert np.abs(base - d).max() > 1e-6


def test_compressed_tokens_are_permuted_through_and_confidence_is_symmetric():
    cfg = MICRO.with_(n_items=3)
    w, inp = setup(cfg=cfg, delta=3)
    perm = np.array([2, 0, 1])
    h1, c1 = oc.future_correction(inp["h_c"], inp["actions"], w, cfg)
    h2, c2 = oc.future_correction(inp["h_c"][perm], inp["actions"], w, cfg)
    np.testing.assert_allclose(h2, h1[perm], rtol=1e-12, atol=1e-14)
    assert c2 == pytest.approx(c1, rel=1e-12, abs=1e-14)


def test_batch_requests_are_independent():
    cfg = MICRO
    w = make_correction_weights(cfg, 9, std=0.5, bias_std=0.3, norm_std=0.3)
    inp = make_correction_inputs(cfg, 10, 3, 4, 2)
    hc = oc.compress_batch(inp["h_vlm"], w, cfg)
    hc1 = oc.compress_batch(inp["h_vlm"][1:2], w, cfg)
    np.testing.assert_array_equal(hc[1], hc1[0])
    hf, conf = oc.correction_batch(inp["h_c"], inp["actions"], w, cfg)
    hf1, conf1 = oc.correction_batch(inp["h_c"][2:], inp["actions"][2:], w, cfg)
    np.testing.assert_array_equal(hf[2], hf1[0])
    assert conf[2] == conf1[0] and conf.shape == (3,)


def test_committed_actions_must_number_1_to_max_delta():
    w, inp = setup(delta=1)
    with pytest.raises(ValueError):
        oc.future_correction(inp["h_c"], inp["actions"][:0], w, MICRO)
    too_many = np.zeros((MICRO.max_delta + 1, MICRO.action_dim))
    with pytest.raises(ValueError):
        oc.future_correction(inp["h_c"], too_many, w, MICRO)


# ---------------------------------------------------------------- the paper's sizes

def test_sizes_match_the_paper():
    path = os.path.join(os.path.dirname(__file__), "golden", "pi05_correction_dims.txt")
    dims = {}
    for line in open(path):
        line = line.split("#")[0].strip()
        if line:
            k, v = (s.strip() for s in line.split("="))
            dims[k] = int(v)
    cfg = PI05_CORRECTION
    assert cfg.n_items == dims["items"]
    assert cfg.width == dims["d_ae"] == PI05.width
    assert cfg.d_vlm == dims["d_vlm"] == GEMMA2B.width
    assert cfg.n_heads * cfg.head_dim == cfg.width
    n = correction_param_count(cfg)
    assert abs(n / 1e6 - dims["params_millions"]) < 0.15 * dims["params_millions"], n
