"""Planted mistakes in a copy of the oracle must each fail at least one pin.

Each mutation is a plausible slip (a dropped term, a wrong sign, index or order, a transposed
operand). The mutated source is loaded as a separate module on the CPU and the pins of
``test_oracle_pins`` are run against it; the real oracle is untouched.
"""

import inspect
import os
import types

import pytest

import tests.test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(os.path.dirname(__file__)), "oracle", "expert.py")

MUTATIONS = [
    ("r * (1.0 + sigma) + beta", "r * sigma + beta"),
    ("/ np.sqrt(F64(D))", ""),
    ("vis[:n_ctx, prefix_len + n_ctx:] = False", "vis[:n_ctx, prefix_len:] = False"),
    ("vis[:n_ctx, prefix_len + n_ctx:] = False", "vis[:1, prefix_len + 1:] = False"),
    ("        h[1:n_ctx] = corr", "        h[1:n_ctx] = 0.5 * corr"),
    ("    n_ctx = 1 + T", "    n_ctx = 1"),
    ("[a * cos - b * sin, b * cos + a * sin]", "[a * cos + b * sin, b * cos - a * sin]"),
    ("/ (half - 1)", "/ half"),
    ("[np.sin(theta), np.cos(theta)]", "[np.cos(theta), np.sin(theta)]"),
    ('h = h + ga * (o @ w["wo"][l].T)', 'h = h + (o @ w["wo"][l].T)'),
    ('h = h + gm * (z @ w["w_down"][l].T)', 'h = h + (z @ w["w_down"][l].T)'),
    ("(y + 0.044715 * y ** 3)", "(y + 0.04715 * y ** 3)"),
    ("delta = 1.0 / num_steps", "delta = 1.0 / (num_steps + 1)"),
    ("np.arange(num_steps, dtype=F64) / num_steps", "(np.arange(num_steps, dtype=F64) + 1) / num_steps"),
    ('c1 = swish(w["time_mlp_in_w"] @ e + w["time_mlp_in_b"])', 'c1 = w["time_mlp_in_w"] @ e + w["time_mlp_in_b"]'),
    ('w["time_mlp_out_w"] @ c1', 'w["time_mlp_out_w"].T @ c1'),
    ("pos = P + np.arange(S)", "pos = np.arange(S)"),
    ("K = np.concatenate([prefix_k[l], k], axis=0)", "K = np.concatenate([k, prefix_k[l]], axis=0)"),
    ('h[n_ctx:] = x @ w["action_in_w"].T + w["action_in_b"]', 'h[n_ctx:] = x @ w["action_in_w"].T'),
    ("vel = u[n_ctx:] @", "vel = u[:-1] @"),
    ("return ma[:W], ma[W:2 * W], ma[2 * W:], mm[:W]", "return ma[W:2 * W], ma[:W], ma[2 * W:], mm[:W]"),
    ("z = gelu_tanh(u @ w[\"w_gate\"][l].T) * (u @ w[\"w_up\"][l].T)",
     "z = gelu_tanh(u @ w[\"w_up\"][l].T) * (u @ w[\"w_gate\"][l].T)"),
    ("np.mean(h * h, axis=-1, keepdims=True) + eps", "np.mean(h * h, axis=-1, keepdims=True)"),
    ("base ** (-2.0 * np.arange(half, dtype=F64) / D)", "base ** (-1.0 * np.arange(half, dtype=F64) / D)"),
    ("scores = scores - scores.max(axis=-1, keepdims=True)", "scores = scores - scores.min(axis=-1, keepdims=True)"),
    ("return z / (1.0 + np.exp(-z))", "return z / (1.0 + np.exp(z))"),
    ("x = x + delta * expert_forward", "x = x - delta * expert_forward"),
    ("u = rms_modulate(h, fm[:W], fm[W:], cfg.rms_eps)", "u = rms_modulate(h, fm[W:], fm[:W], cfg.rms_eps)"),
    ("mm[:W], mm[W:2 * W], mm[2 * W:]", "mm[W:2 * W], mm[:W], mm[2 * W:]"),
    ("u = rms_modulate(h, sm, bm, cfg.rms_eps)", "u = rms_modulate(h, sa, ba, cfg.rms_eps)"),
    ('h[0] = w["state_in_w"] @ s + w["state_in_b"]', 'h[0] = w["state_in_w"] @ s'),
    ('vel = u[n_ctx:] @ w["action_out_w"].T + w["action_out_b"]', 'vel = u[n_ctx:] @ w["action_out_w"].T'),
    ("        k = rope(k, pos, cfg.rope_base)\n", "        k = rope(k, pos, cfg.rope_base)\n        v = rope(v, pos, cfg.rope_base)\n"),
    ("V = np.concatenate([prefix_v[l], v], axis=0)", "V = np.concatenate([prefix_k[l], v], axis=0)"),
]


def _load_mutant(old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, old
    mod = types.ModuleType("oracle_mutant")
    exec(compile(src.replace(old, new), "oracle_mutant", "exec"), mod.__dict__)
    return mod


def _pin_cases():
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        marks = getattr(fn, "pytestmark", [])
        params = [m for m in marks if m.name == "parametrize"]
        if params:
            argname, values = params[0].args
            for v in values:
                yield name, lambda fn=fn, argname=argname, v=v: fn(**{argname: v})
        else:
            yield name, fn


@pytest.mark.parametrize("old,new", MUTATIONS, ids=[f"m{i}" for i in range(len(MUTATIONS))])
def test_mutation_is_caught(old, new, monkeypatch):
    mutant = _load_mutant(old, new)
    monkeypatch.setattr(pins, "oracle", mutant)
    caught = []
    for name, case in _pin_cases():
        try:
            case()
        except Exception:          # an assertion or a shape error: the pin caught the slip
            caught.append(name)
    assert caught, f"no pin catches mutation {old!r} -> {new!r}"
