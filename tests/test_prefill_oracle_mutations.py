"""Planted mistakes in a copy of the LLM-prefill oracle must each fail at least one pin of
tests/test_prefill_oracle_pins.py. The mutated source is loaded as a separate module on the CPU;
the real oracle is untouched."""

import inspect
import os
import types

import pytest

import tests.test_prefill_oracle_pins as pins

SRC = os.path.join(os.path.dirname(os.path.dirname(__file__)), "oracle", "prefill.py")

MUTATIONS = [
    ("visible = np.ones((P, P), dtype=bool)", "visible = np.tril(np.ones((P, P), dtype=bool))"),
    ("        k = rope(k, pos, cfg.rope_base)", "        k = k"),
    ("        v = u @ w[\"wv\"][l].T", "        v = rope(u @ w[\"wv\"][l].T, pos, cfg.rope_base)"),
    ("    pos = np.arange(P)", "    pos = np.arange(P) + 1"),
    ("u = rms_modulate(h, w[\"mlp_norm\"][l], 0.0, cfg.rms_eps)", "u = rms_modulate(h, w[\"attn_norm\"][l], 0.0, cfg.rms_eps)"),
    ("        u = rms_modulate(h, w[\"attn_norm\"][l], 0.0, cfg.rms_eps)   # R17", "        u = h"),
    ("(gelu_tanh(u @ w[\"w_gate\"][l].T) * (u @ w[\"w_up\"][l].T))", "(gelu_tanh(u @ w[\"w_up\"][l].T) * (u @ w[\"w_gate\"][l].T))"),
    ("        return K, V, rms_modulate(h, w[\"final_norm\"], 0.0, cfg.rms_eps)", "        return K, V, h"),
    ("        h = h + o @ w[\"wo\"][l].T", "        h = o @ w[\"wo\"][l].T"),
    ("        o = attention(q, k, v, visible).reshape(P, H * D)", "        o = attention(q, k, k, visible).reshape(P, H * D)"),
    ("        q = rope(q, pos, cfg.rope_base)                            # R18", "        q = q"),
    ("        K[l], V[l] = k, v                                          # R20", "        K[l], V[l] = v, k"),
    ("h = h + (gelu_tanh(u @ w[\"w_gate\"][l].T) * (u @ w[\"w_up\"][l].T)) @ w[\"w_down\"][l].T",
     "h = (gelu_tanh(u @ w[\"w_gate\"][l].T) * (u @ w[\"w_up\"][l].T)) @ w[\"w_down\"][l].T"),
    ("        return K, V, rms_modulate(h, w[\"final_norm\"], 0.0, cfg.rms_eps)",
     "        return K, V, rms_modulate(h, w[\"final_norm\"] - 1.0, 0.0, cfg.rms_eps)"),
    ("        q = (u @ w[\"wq\"][l].T).reshape(P, H, D)", "        q = (u @ w[\"wq\"][l].T).reshape(H, P, D).transpose(1, 0, 2)"),
]


def _load_mutant(old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, old
    mod = types.ModuleType("oracle.prefill_mutant")
    mod.__package__ = "oracle"
    exec(compile(src.replace(old, new), "oracle_prefill_mutant", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("old,new", MUTATIONS, ids=[f"m{i}" for i in range(len(MUTATIONS))])
def test_mutation_is_caught(old, new, monkeypatch):
    mutant = _load_mutant(old, new)
    monkeypatch.setattr(pins, "pf", mutant)
    caught = []
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        try:
            fn()
        except Exception:          # an assertion or a shape error: the pin caught the slip
            caught.append(name)
    assert caught, f"no pin catches mutation {old!r} -> {new!r}"
