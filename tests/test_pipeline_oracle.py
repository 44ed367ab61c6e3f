"""The Jetson-PI control loop composed from the CPU oracles (App. C Alg. 1 over the LLM prefill,
the Q-Former compressor, the future correction module and the action expert's denoise): the
components' widths fit together at the pi0.5 sizes, and the scheduler hands each component the
outputs of the others as Alg. 1 prescribes. CPU only, tiny shapes."""

import numpy as np

import oracle.correction as oc
import oracle.expert as ox
import oracle.prefill as pf
from paper_2607_12659_gb300.scheduler import ConfidenceScheduler
from synth import (GEMMA2B, PI05, PI05_CORRECTION, TINY, make_correction_weights, make_llm_weights,
                   make_prefix_embeddings, make_requests, make_weights)

LLM = GEMMA2B.with_(n_layers=2, width=10, n_heads=2, head_dim=4, mlp_dim=12, precision="fp32")
EXPERT = TINY.with_(n_layers=2, width=8, n_heads=2, head_dim=4, mlp_dim=12, action_dim=3,
                    state_dim=3, time_dim=8)
CORR = PI05_CORRECTION.with_(width=8, n_heads=2, head_dim=4, mlp_dim=12, d_vlm=10, n_items=2,
                             action_dim=3, max_delta=6, precision="fp32")
P, C, N = 5, 6, 2


def test_pi05_component_widths_fit_together():
    # App. A: layer l of the LLM feeds its KV (one head of width D) to layer l of the expert;
    # the compressor reads the LLM's output and the items enter the expert at its width (R15).
    assert PI05.n_layers == GEMMA2B.n_layers and PI05.head_dim == GEMMA2B.head_dim
    assert PI05_CORRECTION.d_vlm == GEMMA2B.width
    assert PI05_CORRECTION.width == PI05.width
    assert PI05_CORRECTION.action_dim == PI05.action_dim
    assert PI05_CORRECTION.max_delta >= 9          # the largest Delta of the results table


class Chain:
    def __init__(self):
        self.wl = pf.to_f64_llm(make_llm_weights(LLM, 1, std=0.3, norm_std=0.2))
        self.wc = oc.to_f64_corr(make_correction_weights(CORR, 2, std=0.3, bias_std=0.2))
        self.we = ox.to_f64(make_weights(EXPERT, 3, std=0.3, bias_std=0.2))
        req = make_requests(EXPERT, 4, 1, P, C)
        self.state, self.noise = req["state"][0].astype(np.float64), req["noise"][0].astype(np.float64)
        self.obs = make_prefix_embeddings(LLM, 5, 2, P).astype(np.float64)
        self.n_obs = 0
        self.log = []

    def observe(self):
        o = self.obs[self.n_obs]
        self.n_obs += 1
        return o

    def vlm(self, x):
        K, V, out = pf.llm_prefill(x, self.wl, LLM, return_output=True)
        h = oc.qformer_compress(out, self.wc, CORR)             # R28
        self.log.append(("vlm", h))
        return h, (K, V)

    def corr(self, h, actions):
        hf, c = oc.future_correction(h, np.array(actions), self.wc, CORR)
        self.log.append(("corr", h, np.array(actions), hf))
        return hf, c

    def act(self, h, kv):
        chunk = ox.denoise(self.noise, self.state, N, kv[0], kv[1], self.we, EXPERT, corr=h)
        self.log.append(("act", h, kv, chunk))
        return list(chunk)


def test_alg1_passes_each_component_the_others_outputs():
    ch = Chain()
    sch = ConfidenceScheduler(vlm=ch.vlm, corr=ch.corr, act=ch.act, observe=ch.observe,
                              theta=-1e30, delta=4, delta_ae=2)
    sch.start()
    _, h0 = ch.log[0]
    K0, V0 = sch.kv
    _, h_act, kv_act, chunk0 = ch.log[1]
    assert h_act is h0 and kv_act[0] is K0
    want = ox.denoise(ch.noise, ch.state, N, K0, V0, ch.we, EXPERT, corr=h0)
    np.testing.assert_array_equal(np.array(sch.buffer.committed(C)), want)

    # Confidence 0 > theta: the VLM is skipped; f_corr sees the state buffer and the next
    # delta_ae committed actions, and the expert runs on its prediction with the old KV.
    assert sch.iterate() == "correction"
    _, h_in, acts_in, hf = ch.log[2]
    assert h_in is h0
    np.testing.assert_array_equal(acts_in, chunk0[:2])
    want_hf, want_c = oc.future_correction(h0, chunk0[:2], ch.wc, CORR)
    np.testing.assert_array_equal(hf, want_hf)
    assert sch.confidence == want_c
    chunk1 = ox.denoise(ch.noise, ch.state, N, K0, V0, ch.we, EXPERT, corr=want_hf)
    np.testing.assert_array_equal(np.array(sch.buffer.committed(2 + C)),
                                  np.concatenate([chunk0[:2], chunk1]))

    # Force the low-confidence branch: a fresh observation through the prefill and the
    # compressor, f_corr over delta committed actions, the expert on the new KV.
    sch.confidence = -1e31
    assert sch.iterate() == "vlm"
    assert ch.n_obs == 2
    K1, V1, out1 = pf.llm_prefill(ch.obs[1], ch.wl, LLM, return_output=True)
    np.testing.assert_array_equal(sch.kv[0], K1)
    committed = np.concatenate([chunk0[:2], chunk1[:2]])
    _, h_in, acts_in, hf2 = ch.log[5]
    np.testing.assert_array_equal(h_in, oc.qformer_compress(out1, ch.wc, CORR))
    np.testing.assert_array_equal(acts_in, committed)
    chunk2 = ox.denoise(ch.noise, ch.state, N, K1, V1, ch.we, EXPERT, corr=hf2)
    np.testing.assert_array_equal(np.array(sch.buffer.committed(4 + C)),
                                  np.concatenate([committed, chunk2]))
    assert np.all(np.isfinite(chunk2))
