"""The correction module's CUDA path (csrc/corr.cu through include/jpi_corr.h) against the fp64
oracle (oracle/correction.py) on the same seeded inputs: the Q-Former compressor, f_corr for
several Delta, the VLM branch's chain, requests alone and inside a batch, the pi0.5-sized
module at batch 1 and 2, and the predicted items handed to the expert on the device.

Tolerance: activations and sums are fp32 and the weights the kernels read are exactly the
oracle's (bf16-representable in bf16 precision), so the differences are fp32 rounding: unit
roundoff 6e-8, grown about sqrt(n) over sums of up to n = 2048 terms (~3e-6 relative) and over
some twenty dependent stages whose LayerNorms rescale by O(1): well inside 5e-4 max-abs and
5e-5 relative L2 on the O(1) outputs. The confidence is held to the same 5e-4.
"""

import numpy as np
import pytest

import oracle
import oracle.correction as oc
from synth import (PI05_CORRECTION, TINY, make_correction_inputs, make_correction_weights,
                   make_requests, make_weights)


pytestmark = pytest.mark.gpu

MAX_ABS, REL_L2 = 5e-4, 5e-5

# Small module that still spans several warps per row, a ragged d_vlm (160 against 256-column
# blocks), a ragged token count and an action width that takes the scalar path.
SMALL = PI05_CORRECTION.with_(width=128, n_heads=4, head_dim=32, mlp_dim=192, d_vlm=160, n_items=4,
                              action_dim=7, max_delta=12, precision="fp32")


def _lib():
    from tests.gpu_util import lib
    lib()
    from paper_2607_12659_gb300 import corr
    return corr


def _close(got, want, what):
    from tests.gpu_util import errors, log_errors
    err, rel = errors(got, want)
    log_errors("correction module: " + what, err, rel)
    assert err <= MAX_ABS and rel <= REL_L2, f"{what}: max-abs {err:.3g}, rel-L2 {rel:.3g}"


def _setup(cfg, seed, B, T, delta, std=0.1, max_batch=4, max_tokens=64):
    import torch
    corr = _lib()
    w = make_correction_weights(cfg, seed, std=std, bias_std=0.1)
    inp = make_correction_inputs(cfg, seed + 1, B, T, delta)
    mod = corr.Corrector(cfg, w, max_batch=max_batch, max_vlm_tokens=max_tokens)
    dev = {k: torch.from_numpy(v).cuda() for k, v in inp.items()}
    return mod, w, inp, dev


# bf16 VLM states are drawn in bf16 precision only, so that pairing has no fp32 case.
@pytest.mark.parametrize("precision,vlm_dtype",
                         [("fp32", "float32"), ("bf16", "float32"), ("bf16", "bfloat16")])
def test_compressor_matches_the_oracle(precision, vlm_dtype):
    import torch
    cfg = SMALL.with_(precision=precision)
    mod, w, inp, dev = _setup(cfg, 11, 3, 45, 5)
    hv = dev["h_vlm"].to(getattr(torch, vlm_dtype))
    got = mod.compress(hv)
    torch.cuda.synchronize()
    want = oc.compress_batch(inp["h_vlm"], w, cfg)
    _close(got.cpu().numpy(), want, "compress")
    mod.close()


@pytest.mark.parametrize("delta", [1, 5, 12])
@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_prediction_matches_the_oracle(delta, precision):
    import torch
    cfg = SMALL.with_(precision=precision)
    mod, w, inp, dev = _setup(cfg, 21, 3, 10, delta)
    hf, conf = mod.predict(dev["h_c"], dev["actions"])
    torch.cuda.synchronize()
    want_h, want_c = oc.correction_batch(inp["h_c"], inp["actions"], w, cfg)
    _close(hf.cpu().numpy(), want_h, "predicted state")
    assert np.abs(conf.cpu().numpy() - want_c).max() <= MAX_ABS
    mod.close()


def test_vlm_branch_chain_and_in_place_feedback():
    import torch
    cfg = SMALL.with_(precision="bf16")
    mod, w, inp, dev = _setup(cfg, 31, 2, 33, 7)
    state = mod.compress(dev["h_vlm"])
    hf, conf = mod.predict(state, dev["actions"], out=state)    # the state buffer fed back in place
    torch.cuda.synchronize()
    w64 = oc.to_f64_corr(w)
    for b in range(2):
        want_h, want_c = oc.correct_from_vlm(inp["h_vlm"][b].astype(np.float64),
                                             inp["actions"][b].astype(np.float64), w64, cfg)
        _close(hf[b].cpu().numpy(), want_h, f"chain request {b}")
        assert abs(float(conf[b]) - want_c) <= MAX_ABS
    mod.close()


def test_a_request_alone_and_inside_a_batch_agree_bit_for_bit():
    import torch
    cfg = SMALL.with_(precision="bf16")
    mod, w, inp, dev = _setup(cfg, 41, 4, 40, 6)
    s4 = mod.compress(dev["h_vlm"])
    h4, c4 = mod.predict(s4, dev["actions"])
    s1 = mod.compress(dev["h_vlm"][2:3])
    h1, c1 = mod.predict(s1, dev["actions"][2:3])
    torch.cuda.synchronize()
    assert torch.equal(s4[2], s1[0]) and torch.equal(h4[2], h1[0]) and torch.equal(c4[2:3], c1)
    mod.close()


@pytest.mark.parametrize("B", [1, 2])
def test_pi05_sized_module(B):
    # d_AE 1024, d_VLM 2048, T' = 4, 816 VLM tokens, Delta = 9 (the largest of the results table).
    import torch
    cfg = PI05_CORRECTION
    mod, w, inp, dev = _setup(cfg, 51, B, 816, 9, std=0.02, max_batch=2, max_tokens=816)
    state = mod.compress(dev["h_vlm"].to(torch.bfloat16))
    hf, conf = mod.predict(state, dev["actions"])
    torch.cuda.synchronize()
    _close(state.cpu().numpy(), oc.compress_batch(inp["h_vlm"], w, cfg), "pi0.5 compress")
    want_h, want_c = oc.correction_batch(state.cpu().numpy().astype(np.float64), inp["actions"], w, cfg)
    _close(hf.cpu().numpy(), want_h, "pi0.5 predict")
    assert np.abs(conf.cpu().numpy() - want_c).max() <= MAX_ABS
    mod.close()


def test_predicted_items_drive_the_expert_on_the_device():
    # f_corr's output goes to jpi_set_correction without leaving the GPU; the expert's denoise
    # with those items matches the oracle's denoise with the same items.
    import torch
    from tests.gpu_util import make_expert
    ecfg = TINY
    cfg = SMALL.with_(width=ecfg.width, n_heads=4, head_dim=64, action_dim=ecfg.action_dim, precision="fp32")
    mod, w, inp, dev = _setup(cfg, 61, 2, 20, 4)
    items, _ = mod.predict(dev["h_c"], dev["actions"])
    we = make_weights(ecfg, 62)
    P, C, N = 16, 8, 3
    r = make_requests(ecfg, 63, 2, P, C)
    ex = make_expert(ecfg, we, max_batch=2, max_prefix=P, max_chunk=C, max_steps=N)
    ex.set_prefix_kv(torch.from_numpy(r["prefix_k"]).cuda(), torch.from_numpy(r["prefix_v"]).cuda())
    ex.set_correction(items)
    out = ex.denoise(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), N)
    torch.cuda.synchronize()
    want = oracle.denoise_batch(r["noise"], r["state"], N, r["prefix_k"], r["prefix_v"], we, ecfg,
                                corr=items.cpu().numpy())
    assert np.abs(out.cpu().numpy() - want).max() <= 1e-4
    ex.close()
    mod.close()


def test_alg1_on_the_gpu_components():
    # Alg. 1 with f_corr and the compressor from the library and the expert as f_act: each chunk
    # is the expert's denoise for the state the module predicted from the compressed VLM output.
    import torch
    from paper_2607_12659_gb300.scheduler import (ConfidenceScheduler, corrector_corr, corrector_vlm,
                                                  expert_act)
    from tests.gpu_util import make_expert
    ecfg = TINY
    cfg = SMALL.with_(width=ecfg.width, n_heads=4, head_dim=64, action_dim=ecfg.action_dim, precision="fp32")
    mod, w, inp, dev = _setup(cfg, 71, 1, 24, 4, max_batch=1)
    we = make_weights(ecfg, 72)
    P, C, N = 16, 8, 3
    r = make_requests(ecfg, 73, 1, P, C)
    ex = make_expert(ecfg, we, max_batch=1, max_prefix=P, max_chunk=C, max_steps=N)
    kv = (torch.from_numpy(r["prefix_k"]).cuda(), torch.from_numpy(r["prefix_v"]).cuda())
    state = torch.from_numpy(r["state"]).cuda()
    noise = torch.from_numpy(r["noise"]).cuda()
    sch = ConfidenceScheduler(vlm=corrector_vlm(lambda obs: (dev["h_vlm"], kv), mod), corr=corrector_corr(mod),
                              act=expert_act(ex, lambda: state, lambda: noise, N), observe=lambda: "obs",
                              theta=-1e30, delta=4, delta_ae=2)
    sch.start()
    first = np.stack(sch.buffer.committed(C))
    sch.iterate()
    torch.cuda.synchronize()
    w64 = oc.to_f64_corr(w)
    h0 = oc.qformer_compress(inp["h_vlm"][0].astype(np.float64), w64, cfg)
    h1, c1 = oc.future_correction(h0, first[:2].astype(np.float64), w64, cfg)
    assert abs(sch.confidence - c1) <= MAX_ABS
    want = oracle.denoise_batch(r["noise"], r["state"], N, r["prefix_k"], r["prefix_v"], we, ecfg,
                                corr=h1[None])
    got = np.stack(sch.buffer.committed(2 + C))[2:]
    assert np.abs(got - want[0]).max() <= 1e-3
    ex.close()
    mod.close()


def test_alg1_with_every_component_on_the_gpu():
    # Prefill (KV straight into the expert's store) -> compressor -> expert at start-up, then
    # f_corr -> expert: the first chunk against the oracles' chain.
    import torch
    import oracle.prefill as pf
    from paper_2607_12659_gb300 import prefill
    from paper_2607_12659_gb300.scheduler import (ConfidenceScheduler, corrector_corr, corrector_vlm,
                                                  expert_act, prefill_vlm)
    from synth import GEMMA2B, PI05, make_llm_weights, make_prefix_embeddings
    from tests.gpu_util import make_expert
    ecfg = PI05.with_(n_layers=2, width=256, n_heads=2, head_dim=128, mlp_dim=512, time_dim=64)   # bf16 store
    lcfg = GEMMA2B.with_(n_layers=2, width=192, n_heads=2, head_dim=128, mlp_dim=384, precision="fp32")
    cfg = SMALL.with_(width=256, n_heads=4, head_dim=64, d_vlm=192, action_dim=ecfg.action_dim)
    P, C, N = 24, 8, 3
    wl = make_llm_weights(lcfg, 91, std=0.05)
    wc = make_correction_weights(cfg, 92, std=0.1, bias_std=0.1)
    we = make_weights(ecfg, 93)
    x = make_prefix_embeddings(lcfg, 94, 1, P)
    r = make_requests(ecfg, 95, 1, 1, C)
    pre = prefill.Prefill(lcfg, wl, max_batch=1, max_prefix=P)
    mod = _lib().Corrector(cfg, wc, max_batch=1, max_vlm_tokens=P)
    ex = make_expert(ecfg, we, max_batch=1, max_prefix=P, max_chunk=C, max_steps=N)
    state, noise = torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda()
    vlm = corrector_vlm(prefill_vlm(pre, ex, lambda obs: torch.from_numpy(x).cuda()), mod)
    sch = ConfidenceScheduler(vlm=vlm, corr=corrector_corr(mod),
                              act=expert_act(ex, lambda: state, lambda: noise, N, set_kv=lambda *kv: None),
                              observe=lambda: "obs", theta=-1e30, delta=4, delta_ae=2)
    sch.start()
    torch.cuda.synchronize()
    first = np.stack(sch.buffer.committed(C))
    K, V, out = pf.prefill_batch(x, wl, lcfg)
    h0 = oc.compress_batch(out.astype(np.float32), wc, cfg)
    want = oracle.denoise_batch(r["noise"], r["state"], N, K.astype(np.float32), V.astype(np.float32), we, ecfg,
                                corr=h0)
    # bf16 GEMM operands in the prefill, then the bf16 expert on the KV it wrote.
    assert np.abs(first - want[0]).max() <= 5e-2
    ex.close()
    mod.close()
    pre.close()
