"""Confidence-based scheduling of Jetson-PI (App. C, Alg. 1): when to rerun the VLM.

Host control logic around the action expert. The VLM, the future correction module and the
observation source are callables supplied by the caller (they are outside this library); the
action expert is usually `expert_act(...)`, which runs the expert's flow-matching denoise on the
GPU with the predicted compressed VLM state as correction items; `corrector_corr` and
`corrector_vlm` build f_corr and the compressing side of f_vlm from the library's correction
module (`corr.Corrector`).

One iteration, after the start-up pass (VLM on the first observation, expert on its output):
  * confidence c > theta (theta < 0): skip the VLM. Take the next delta_ae actions of the
    buffer (they run while the expert works), let the correction module predict the VLM state
    at t + delta_ae from the last state in the state buffer, and refill the action buffer from
    t + delta_ae with the expert's chunk for that state and the KV buffer.
  * otherwise: observe, take the next delta actions, run the VLM (refreshing the KV buffer),
    predict the state at t + delta from the fresh one, refill from t + delta.
The new confidence comes from the correction module each time. The initial confidence is 0, so
the first iteration after start-up skips the VLM (Alg. 1 initialises it as a large confidence).

Actions are indexed by control step. `ActionBuffer` is what an executor thread consumes
(`pop`) while the scheduler refills it (`replace_from`); the scheduler advances t by what was
executed meanwhile. The new chunk starts right after the committed actions f_corr was given:
t + delta_ae (or t + delta) while the buffer holds that many, earlier when it holds fewer, so
the executor, which stops at the first empty control step, always reaches it.
"""

from __future__ import annotations

import threading
from dataclasses import dataclass, field
from typing import Any, Callable, Sequence

import numpy as np


class ActionBuffer:
    """Actions keyed by control step; thread-safe. The executor pops the action of the current
    step; the scheduler replaces everything from a given step on with a new chunk."""

    def __init__(self):
        self._lock = threading.Lock()
        self._next = 0          # control step of the next action to execute
        self._actions = {}      # step -> action

    @property
    def next_step(self) -> int:
        with self._lock:
            return self._next

    def replace_from(self, step: int, chunk: Sequence[Any]) -> None:
        """Drop every action at or after `step` and store `chunk[k]` at step + k. Steps the
        executor has already passed (it kept running while the chunk was computed) are not
        stored: their time is gone."""
        with self._lock:
            for s in [s for s in self._actions if s >= step]:
                del self._actions[s]
            for k, a in enumerate(chunk):
                if step + k >= self._next:
                    self._actions[step + k] = a

    def committed(self, n: int) -> list:
        """The next n actions to be executed (those the robot runs while inference is in
        flight); fewer if the buffer holds fewer."""
        with self._lock:
            out = []
            for s in range(self._next, self._next + n):
                if s not in self._actions:
                    break
                out.append(self._actions[s])
            return out

    def pop(self):
        """The action of the current control step (None if the buffer ran dry), advancing it."""
        with self._lock:
            a = self._actions.pop(self._next, None)
            if a is not None:
                self._next += 1
            return a

    def __len__(self) -> int:
        with self._lock:
            return sum(1 for s in self._actions if s >= self._next)


@dataclass
class SchedulerTrace:
    """What each iteration did: 'start', 'correction' (VLM skipped) or 'vlm'."""
    branch: str
    t: int
    confidence_before: float
    confidence_after: float
    committed: int


@dataclass
class ConfidenceScheduler:
    """Alg. 1 of App. C.

    vlm(obs) -> (h, kv): the VLM's compressed final-layer state and its per-layer KV.
    corr(h, actions) -> (h_future, confidence): the future correction module.
    act(h, kv) -> chunk: the action expert (a sequence of actions).
    observe() -> obs.
    theta < 0: confidence threshold; delta / delta_ae: VLA and expert latency in actions.
    """
    vlm: Callable[[Any], tuple]
    corr: Callable[[Any, list], tuple]
    act: Callable[[Any, Any], Sequence[Any]]
    observe: Callable[[], Any]
    theta: float
    delta: int
    delta_ae: int
    buffer: ActionBuffer = field(default_factory=ActionBuffer)
    trace: list = field(default_factory=list)

    def __post_init__(self):
        if not self.theta < 0.0:
            raise ValueError("theta must be negative (App. C)")
        if self.delta < 1 or self.delta_ae < 1:
            raise ValueError("delta and delta_ae must be >= 1 action")
        self.t = 0
        self.confidence = 0.0
        self.h = None    # state buffer B_h
        self.kv = None   # KV buffer B_kv
        self.started = False

    def start(self) -> None:
        """Initial VLM pass on the first observation and the first chunk at step 0."""
        h0, kv0 = self.vlm(self.observe())
        self.h, self.kv = h0, kv0
        self.buffer.replace_from(self.buffer.next_step, self.act(h0, kv0))
        self.confidence = 0.0
        self.t = self.buffer.next_step
        self.started = True
        self.trace.append(SchedulerTrace("start", self.t, 0.0, 0.0, 0))

    def iterate(self) -> str:
        """One pass of the loop body; returns the branch taken."""
        if not self.started:
            raise RuntimeError("call start() first")
        c0 = self.confidence
        t = self.buffer.next_step    # actions executed so far advance t
        if c0 > self.theta:
            committed = self.buffer.committed(self.delta_ae)
            h_future, c = self.corr(self.h, committed)
            chunk = self.act(h_future, self.kv)
            self.buffer.replace_from(t + len(committed), chunk)
            branch = "correction"
        else:
            obs = self.observe()
            committed = self.buffer.committed(self.delta)
            h_t, kv_t = self.vlm(obs)
            self.kv = kv_t
            h_future, c = self.corr(h_t, committed)
            chunk = self.act(h_future, self.kv)
            self.buffer.replace_from(t + len(committed), chunk)
            branch = "vlm"
        self.h = h_future
        self.confidence = float(c)
        self.t = t
        self.trace.append(SchedulerTrace(branch, t, c0, self.confidence, len(committed)))
        return branch


def expert_act(expert, state_fn: Callable[[], Any], noise_fn: Callable[[], Any], num_steps: int,
               set_kv: Callable[[Any, Any], None] | None = None):
    """f_act over the library: the correction items h ([B][T'][width] CUDA tensor) go in as
    context tokens, the KV buffer is (re)loaded when it changes, and the flow-matching denoise
    returns the chunk ([B][C][A], as a host array)."""
    last = {"kv": None}

    def act(h, kv):
        if kv is not last["kv"]:
            if set_kv is not None:
                set_kv(*kv)
            else:
                expert.set_prefix_kv(*kv)
            last["kv"] = kv
        expert.set_correction(h)
        out = expert.denoise(state_fn(), noise_fn(), num_steps)
        return out.cpu().numpy()[0]
    return act


def corrector_corr(corrector):
    """f_corr over the library's correction module: the state buffer holds a compressed state
    ([1][T'][width] CUDA tensor) and the committed actions are the executor's action rows; returns
    the predicted state (on the device) and its confidence (one host float, read back because the
    scheduler branches on it).

    With no committed action (the executor ran the buffer dry) there is nothing to predict ahead:
    the state passes through with confidence 0, the value Alg. 1 starts from. More committed
    actions than the module's position table holds is an error."""
    import torch

    def corr(h, actions):
        if len(actions) == 0:
            return h, 0.0
        if len(actions) > corrector.dims.max_delta:
            raise ValueError(f"{len(actions)} committed actions exceed the correction module's "
                             f"max_delta {corrector.dims.max_delta}")
        a = torch.as_tensor(np.stack([np.asarray(x, np.float32) for x in actions])[None],
                            device=h.device)
        h_future, conf = corrector.predict(h, a)
        return h_future, float(conf[0].item())
    return corr


def corrector_vlm(vlm_forward, corrector):
    """f_vlm followed by the compressor (Alg. 1's state buffer holds compressed states):
    vlm_forward(obs) -> (final-layer output [1][T][d_VLM] CUDA tensor, kv)."""
    def vlm(obs):
        out, kv = vlm_forward(obs)
        return corrector.compress(out), kv
    return vlm


def prefill_vlm(prefill, expert, embed: Callable[[Any], Any]):
    """f_vlm's language-model part over the library: embed(obs) gives the prefix token
    embeddings [1][P][W] (CUDA); the prefill writes every layer's keys and values straight into
    the expert's store and commits it, and returns the final-layer output. The KV handle it
    returns is a fresh token, so pair it with expert_act(..., set_kv=lambda *kv: None): the store
    is already current."""
    count = [0]

    def vlm(obs):
        out = prefill.into_expert(embed(obs), expert)
        count[0] += 1
        return out, (count[0],)
    return vlm
