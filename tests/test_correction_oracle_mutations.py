"""Planted mistakes in a copy of the future-correction oracle must each fail at least one pin of
tests/test_correction_oracle_pins.py. The mutated source is loaded as a separate module on the
CPU; the real oracle is untouched."""

import inspect
import os
import types

import pytest

import tests.test_correction_oracle_pins as pins

SRC = os.path.join(os.path.dirname(os.path.dirname(__file__)), "oracle", "correction.py")

MUTATIONS = [
    # LayerNorm: unbiased variance, a dropped shift.
    ("var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)", "var = x.var(axis=-1, ddof=1, keepdims=True)"),
    ("return (x - mu) / np.sqrt(var + eps) * w + b", "return x / np.sqrt(var + eps) * w + b"),
    # attention: no scale, softmax over queries, heads and rows mixed, dropped q / v / o biases.
    ("scores = np.einsum(\"ihd,jhd->hij\", q, k) / np.sqrt(F64(Dh))", "scores = np.einsum(\"ihd,jhd->hij\", q, k)"),
    ("pr = pr / pr.sum(axis=-1, keepdims=True)", "pr = pr / pr.sum(axis=-2, keepdims=True)"),
    ("o = np.einsum(\"hij,jhd->ihd\", pr, v).reshape(n, H * Dh)", "o = np.einsum(\"hij,jhd->hid\", pr, v).reshape(n, H * Dh)"),
    ("q = (xq @ w[p + \"wq\"].T + w[p + \"bq\"]).reshape(n, H, Dh)", "q = (xq @ w[p + \"wq\"].T).reshape(n, H, Dh)"),
    ("v = (xkv @ w[p + \"wv\"].T + w[p + \"bv\"]).reshape(m, H, Dh)", "v = (xkv @ w[p + \"wv\"].T).reshape(m, H, Dh)"),
    ("    return o @ w[p + \"wo\"].T + w[p + \"bo\"]", "    return o @ w[p + \"wo\"].T"),
    # MLP and block.
    ("return gelu_tanh(x @ w[p + \"w1\"].T + w[p + \"b1\"]) @ w[p + \"w2\"].T + w[p + \"b2\"]",
     "return np.maximum(x @ w[p + \"w1\"].T + w[p + \"b1\"], 0.0) @ w[p + \"w2\"].T + w[p + \"b2\"]"),
    ("    return x + mlp(u, w, p + \"mlp_\")", "    return mlp(u, w, p + \"mlp_\")"),
    ("    x = x + multi_head_attention(u, u, w, p + \"sa_\", cfg)", "    x = x + multi_head_attention(x, x, w, p + \"sa_\", cfg)"),
    # Q-Former.
    ("    x = x + multi_head_attention(u, u, w, \"qf_sa_\", cfg)", "    x = x"),
    ("    u = layer_norm(x, w[\"qf_ln2_w\"], w[\"qf_ln2_b\"], cfg.ln_eps)", "    u = x"),
    ("    x = x + multi_head_attention(u, h_vlm, w, \"qf_ca_\", cfg)", "    x = multi_head_attention(u, h_vlm, w, \"qf_ca_\", cfg)"),
    ("    return layer_norm(x, w[\"qf_lnf_w\"], w[\"qf_lnf_b\"], cfg.ln_eps)", "    return x"),
    # action branch.
    ("    x = x + w[\"act_pos\"][:n]", "    x = x + w[\"act_pos\"][1:n + 1]"),
    ("    return x[n - 1]", "    return x[0]"),
    ("x = gelu_tanh(actions @ w[\"act_w1\"].T + w[\"act_b1\"]) @ w[\"act_w2\"].T + w[\"act_b2\"]",
     "x = gelu_tanh(actions @ w[\"act_w1\"].T + w[\"act_b1\"]) @ w[\"act_w2\"].T"),
    ("    x = transformer_block(x, w, \"ab_\", cfg)", "    x = x"),
    # join, joint blocks, heads.
    ("joined = np.concatenate([h_c, np.broadcast_to(s, h_c.shape)], axis=-1)",
     "joined = np.concatenate([np.broadcast_to(s, h_c.shape), h_c], axis=-1)"),
    ("    for i in range(cfg.n_joint):", "    for i in range(cfg.n_joint - 1):"),
    ("        x = transformer_block(x, w, f\"jb{i}_\", cfg)", "        x = transformer_block(x, w, \"jb0_\", cfg)"),
    ("    h_future = u @ w[\"corr_w\"].T + w[\"corr_b\"]", "    h_future = u @ w[\"corr_w\"].T + w[\"corr_b\"] + h_c"),
    ("confidence = float(w[\"conf_w\"][0] @ u.mean(axis=0) + w[\"conf_b\"][0])",
     "confidence = float(w[\"conf_w\"][0] @ u[0] + w[\"conf_b\"][0])"),
    ("confidence = float(w[\"conf_w\"][0] @ u.mean(axis=0) + w[\"conf_b\"][0])",
     "confidence = float(w[\"conf_w\"][0] @ x.mean(axis=0) + w[\"conf_b\"][0])"),
    ("    return future_correction(qformer_compress(h_vlm, w, cfg), actions, w, cfg)",
     "    return future_correction(h_vlm[:cfg.n_items, :cfg.width], actions, w, cfg)"),
    ("    x = x + w[\"act_pos\"][:n]", "    x = x"),
    ("return (x - mu) / np.sqrt(var + eps) * w + b", "return (x - mu) / np.sqrt(var) * w + b"),
    ("    for i in range(cfg.n_joint):", "    for i in reversed(range(cfg.n_joint)):"),
    ("confidence = float(w[\"conf_w\"][0] @ u.mean(axis=0) + w[\"conf_b\"][0])",
     "confidence = float(w[\"conf_w\"][0] @ u.mean(axis=0))"),
    ("    x = x + mlp(u, w, \"qf_mlp_\")", "    x = mlp(u, w, \"qf_mlp_\")"),
    ("x = gelu_tanh(actions @ w[\"act_w1\"].T + w[\"act_b1\"]) @ w[\"act_w2\"].T + w[\"act_b2\"]",
     "x = (actions @ w[\"act_w1\"].T + w[\"act_b1\"]) @ w[\"act_w2\"].T + w[\"act_b2\"]"),
]


def _load_mutant(old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, old
    mod = types.ModuleType("oracle.correction_mutant")
    mod.__package__ = "oracle"
    exec(compile(src.replace(old, new), "oracle_correction_mutant", "exec"), mod.__dict__)
    return mod


def _pins():
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        marks = getattr(fn, "pytestmark", [])
        params = [m for m in marks if m.name == "parametrize"]
        if params:
            argname, values = params[0].args
            for v in values:
                yield name, (lambda fn=fn, argname=argname, v=v: fn(**{argname: v}))
        else:
            yield name, fn


@pytest.mark.parametrize("old,new", MUTATIONS, ids=[f"m{i}" for i in range(len(MUTATIONS))])
def test_mutation_is_caught(old, new, monkeypatch):
    mutant = _load_mutant(old, new)
    monkeypatch.setattr(pins, "oc", mutant)
    caught = []
    for name, fn in _pins():
        try:
            fn()
        except Exception:          # an assertion or a shape error: the pin caught the slip
            caught.append(name)
    assert caught, f"no pin catches mutation {old!r} -> {new!r}"


def test_the_unmutated_oracle_passes_every_pin():
    for name, fn in _pins():
        fn()
