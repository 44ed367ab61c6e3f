"""Alg. 1 (App. C) confidence-based scheduling, with scripted stand-ins for the VLM, the
correction module and the expert: which components run in each branch, with which inputs, and
where each new chunk lands in the action buffer. CPU only."""

import threading

import pytest

from paper_2607_12659_gb300.scheduler import ActionBuffer, ConfidenceScheduler


class Script:
    """Stand-ins that record their calls. The VLM returns ('h', n) and ('kv', n) for its n-th
    call; corr returns ('hf', m) with the next scripted confidence; act returns a chunk of
    C actions ('a', k, j)."""

    def __init__(self, confidences, C=8):
        self.calls = []
        self.conf = list(confidences)
        self.C = C
        self.nv = self.nc = self.na = self.no = 0

    def observe(self):
        self.no += 1
        self.calls.append(("observe", self.no))
        return ("obs", self.no)

    def vlm(self, obs):
        self.nv += 1
        self.calls.append(("vlm", obs))
        return ("h", self.nv), ("kv", self.nv)

    def corr(self, h, actions):
        self.nc += 1
        self.calls.append(("corr", h, list(actions)))
        return ("hf", self.nc), self.conf.pop(0)

    def act(self, h, kv):
        self.na += 1
        self.calls.append(("act", h, kv))
        return [("a", self.na, j) for j in range(self.C)]


def make(script, theta=-0.2, delta=6, delta_ae=2):
    return ConfidenceScheduler(vlm=script.vlm, corr=script.corr, act=script.act,
                               observe=script.observe, theta=theta, delta=delta, delta_ae=delta_ae)


def test_start_runs_the_vlm_then_the_expert_on_its_state():
    s = Script([])
    sch = make(s)
    sch.start()
    assert s.calls == [("observe", 1), ("vlm", ("obs", 1)), ("act", ("h", 1), ("kv", 1))]
    assert sch.buffer.committed(8) == [("a", 1, j) for j in range(8)]
    assert sch.confidence == 0.0


def test_initial_confidence_skips_the_vlm_and_predicts_delta_ae_ahead():
    s = Script([0.5])
    sch = make(s)
    sch.start()
    s.calls.clear()
    assert sch.iterate() == "correction"
    # corr sees the state buffer and the delta_ae actions that run meanwhile; the expert uses
    # the predicted state with the unchanged KV buffer.
    assert s.calls == [("corr", ("h", 1), [("a", 1, 0), ("a", 1, 1)]),
                       ("act", ("hf", 1), ("kv", 1))]
    # The new chunk starts at step t + delta_ae = 2; steps 0, 1 keep the committed actions.
    assert sch.buffer.committed(4) == [("a", 1, 0), ("a", 1, 1), ("a", 2, 0), ("a", 2, 1)]
    assert sch.h == ("hf", 1) and sch.confidence == 0.5


def test_low_confidence_refreshes_the_vlm_and_predicts_delta_ahead():
    s = Script([-0.5, 0.1, 0.3])
    sch = make(s, delta=3, delta_ae=1)
    sch.start()
    assert sch.iterate() == "correction"          # confidence 0 > theta
    s.calls.clear()
    assert sch.iterate() == "vlm"                 # -0.5 <= theta
    committed = [("a", 1, 0), ("a", 2, 0), ("a", 2, 1)]
    assert s.calls == [("observe", 2), ("vlm", ("obs", 2)), ("corr", ("h", 2), committed),
                       ("act", ("hf", 2), ("kv", 2))]
    assert sch.kv == ("kv", 2)
    assert sch.buffer.committed(5) == committed + [("a", 3, 0), ("a", 3, 1)]
    assert sch.iterate() == "correction"          # 0.1 > theta: the VLM is skipped again
    assert s.calls[-1] == ("act", ("hf", 3), ("kv", 2))


def test_executed_actions_advance_t():
    s = Script([0.3, 0.3])
    sch = make(s, delta=4, delta_ae=2)
    sch.start()
    for _ in range(3):
        sch.buffer.pop()
    sch.iterate()
    assert sch.t == 3
    assert s.calls[-2] == ("corr", ("h", 1), [("a", 1, 3), ("a", 1, 4)])
    assert sch.buffer.committed(3) == [("a", 1, 3), ("a", 1, 4), ("a", 2, 0)]
    assert sch.trace[-1].branch == "correction" and sch.trace[-1].committed == 2


def test_action_buffer_replace_commit_pop():
    b = ActionBuffer()
    b.replace_from(0, [1, 2, 3, 4])
    assert b.committed(2) == [1, 2] and len(b) == 4
    assert b.pop() == 1 and b.next_step == 1
    b.replace_from(2, [30, 40, 50])
    assert b.committed(10) == [2, 30, 40, 50]
    for want in (2, 30, 40, 50):
        assert b.pop() == want
    assert b.pop() is None and b.next_step == 5 and len(b) == 0


def test_executor_thread_and_scheduler_share_the_buffer():
    s = Script([0.5] * 50, C=6)
    sch = make(s, delta=3, delta_ae=2)
    sch.start()
    popped, stop = [], threading.Event()

    def executor():
        while not stop.is_set():
            a = sch.buffer.pop()
            if a is not None:
                popped.append(a)

    th = threading.Thread(target=executor)
    th.start()
    for _ in range(50):
        sch.iterate()
    stop.set()
    th.join()
    # Steps run in order with no gaps, and every action executed came from some chunk.
    assert sch.buffer.next_step == len(popped)
    assert all(a[0] == "a" for a in popped)


def test_theta_must_be_negative():
    with pytest.raises(ValueError):
        make(Script([]), theta=0.1)
    with pytest.raises(RuntimeError):
        make(Script([])).iterate()


def test_library_f_corr_handles_an_empty_buffer_and_too_many_actions():
    # The glue over the correction module, with a stand-in module that records its inputs.
    torch = pytest.importorskip("torch")
    import numpy as np
    from types import SimpleNamespace
    from paper_2607_12659_gb300.scheduler import corrector_corr

    seen = []

    class Stub:
        dims = SimpleNamespace(max_delta=3)

        def predict(self, h, a):
            seen.append(a.shape)
            return h + 1.0, torch.tensor([-0.5])

    corr = corrector_corr(Stub())
    h = torch.zeros(1, 2, 4)
    h2, c = corr(h, [])
    assert h2 is h and c == 0.0 and not seen            # nothing to predict ahead
    h3, c = corr(h, [np.ones(5), np.zeros(5)])
    assert seen == [(1, 2, 5)] and c == -0.5 and float(h3[0, 0, 0]) == 1.0
    with pytest.raises(ValueError):
        corr(h, [np.ones(5)] * 4)


def test_a_short_buffer_puts_the_new_chunk_right_after_what_is_committed():
    # Only one action is left when delta_ae = 3 would be committed: the prediction covers that
    # one action and the new chunk starts right after it, so the executor never stalls on an
    # empty control step.
    s = Script([0.5, 0.5], C=4)
    sch = make(s, delta=6, delta_ae=3)
    sch.start()
    for _ in range(3):
        sch.buffer.pop()                              # steps 0..2 executed, step 3 left
    assert sch.iterate() == "correction"
    assert s.calls[-2] == ("corr", ("h", 1), [("a", 1, 3)])
    assert sch.buffer.committed(5) == [("a", 1, 3), ("a", 2, 0), ("a", 2, 1), ("a", 2, 2), ("a", 2, 3)]
    popped = [sch.buffer.pop() for _ in range(5)]
    assert popped[-1] == ("a", 2, 3) and sch.buffer.next_step == 8


def test_a_chunk_that_arrives_late_keeps_only_its_future_steps():
    b = ActionBuffer()
    b.replace_from(0, [1, 2, 3, 4, 5])
    for _ in range(3):
        b.pop()                                       # steps 0..2 ran while the chunk was computed
    b.replace_from(1, [20, 30, 40, 50])               # meant for steps 1..4
    assert b.committed(3) == [40, 50] and len(b) == 2
    assert b.pop() == 40 and b.pop() == 50 and b.pop() is None
    assert len(b._actions) == 0                       # nothing stale left behind
