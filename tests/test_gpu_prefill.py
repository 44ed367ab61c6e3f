"""The LLM prefill's CUDA path (libjpi_prefill.so through include/jpi_prefill.h) against the fp64
oracle (oracle/prefill.py) on the same seeded inputs: every layer's K and V and the final output
at small shapes (ragged prefix, several requests), two Gemma-2B-sized layers, and the zero-copy
path into the expert's KV store.

Tolerance: every GEMM operand is rounded to bf16 (the normed input, q and K after rotary
coding, V, the probabilities, the attention output, the GeGLU output), each a relative 2^-9 per
element, with fp32 sums and an fp32 residual stream; the K and V written are bf16 themselves.
After a few layers that is about 1% in relative L2, so the tests allow 2e-2 relative L2 and a
max-abs of 5e-2 times the largest reference magnitude.
"""

import numpy as np
import pytest

import oracle.prefill as pf
from synth import GEMMA2B, PI05, make_llm_weights, make_prefix_embeddings, make_requests, make_weights


pytestmark = pytest.mark.gpu

REL_L2, MAX_ABS_FRAC = 2e-2, 5e-2
SMALL = GEMMA2B.with_(n_layers=3, width=256, n_heads=4, head_dim=64, mlp_dim=512, precision="bf16")


def _mods():
    from tests.gpu_util import lib
    lib()
    from paper_2607_12659_gb300 import prefill
    return prefill


def _close(got, want, what):
    from tests.gpu_util import errors, log_errors
    err, rel = errors(got, want)
    log_errors("prefill: " + what, err, rel)
    lim = MAX_ABS_FRAC * float(np.abs(want).max())
    assert rel <= REL_L2 and err <= lim, f"{what}: max-abs {err:.3g} (limit {lim:.3g}), rel-L2 {rel:.3g}"


@pytest.mark.parametrize("B,P,x_dtype", [(1, 64, "float32"), (3, 45, "bfloat16")])
def test_prefill_matches_the_oracle(B, P, x_dtype):
    import torch
    prefill = _mods()
    cfg = SMALL
    w = make_llm_weights(cfg, 81, std=0.05, norm_std=0.1)
    x = make_prefix_embeddings(cfg, 82, B, P)
    pre = prefill.Prefill(cfg, w, max_batch=4, max_prefix=80)
    K, V, out = pre.into_tensors(torch.from_numpy(x).cuda().to(getattr(torch, x_dtype)))
    torch.cuda.synchronize()
    pre.device_status()
    Kw, Vw, want = pf.prefill_batch(x, w, cfg)
    for l in range(cfg.n_layers):
        _close(K[l].float().cpu().numpy(), Kw[l], f"K layer {l}")
        _close(V[l].float().cpu().numpy(), Vw[l], f"V layer {l}")
    _close(out.cpu().numpy(), want, "final output")
    pre.close()


def test_split_products_and_padded_gate_up():
    # H D = 1024 and F = 1096 give the output and down products 16 and 18 k-blocks over few
    # tiles, so both run split over K (partials added to the residual with the next norm), and
    # F is not a multiple of 128, so the last gate/up tile is zero-padded. Without the final
    # output the last split only updates the residual; K and V must not change.
    import torch
    prefill = _mods()
    cfg = GEMMA2B.with_(n_layers=2, width=256, n_heads=4, head_dim=256, mlp_dim=1096)
    w = make_llm_weights(cfg, 91, std=0.05, norm_std=0.1)
    x = make_prefix_embeddings(cfg, 92, 2, 50)
    pre = prefill.Prefill(cfg, w, max_batch=2, max_prefix=50)
    xt = torch.from_numpy(x).cuda()
    K, V, out = pre.into_tensors(xt)
    K2, V2, _ = pre.into_tensors(xt, final=False)
    torch.cuda.synchronize()
    pre.device_status()
    Kw, Vw, want = pf.prefill_batch(x, w, cfg)
    for l in range(cfg.n_layers):
        _close(K[l].float().cpu().numpy(), Kw[l], f"split K layer {l}")
        _close(V[l].float().cpu().numpy(), Vw[l], f"split V layer {l}")
        assert torch.equal(K[l], K2[l]) and torch.equal(V[l], V2[l])
    _close(out.cpu().numpy(), want, "split final output")
    pre.close()


def test_gemma2b_sized_layers():
    # Width 2048, 8 heads x 256, GeGLU 16384, 816 prefix tokens; two layers keep the fp64 oracle
    # to seconds.
    import torch
    prefill = _mods()
    cfg = GEMMA2B.with_(n_layers=2)
    w = make_llm_weights(cfg, 83)
    x = make_prefix_embeddings(cfg, 84, 1, 816)
    pre = prefill.Prefill(cfg, w, max_batch=1, max_prefix=816)
    K, V, out = pre.into_tensors(torch.from_numpy(x).cuda().to(torch.bfloat16))
    torch.cuda.synchronize()
    pre.device_status()
    Kw, Vw, want = pf.prefill_batch(x, w, cfg)
    for l in range(cfg.n_layers):
        _close(K[l].float().cpu().numpy(), Kw[l], f"Gemma-2B K layer {l}")
        _close(V[l].float().cpu().numpy(), Vw[l], f"Gemma-2B V layer {l}")
    _close(out.cpu().numpy(), want, "Gemma-2B final output")
    pre.close()


def test_zero_copy_into_the_expert_store():
    # The prefill writes straight into the expert's KV store; the denoise that follows equals the
    # denoise after copying the same K and V in with jpi_set_prefix_kv, bit for bit.
    import torch
    from tests.gpu_util import make_expert
    prefill = _mods()
    ecfg = PI05.with_(n_layers=2, width=256, n_heads=2, head_dim=128, mlp_dim=512, time_dim=64)
    cfg = GEMMA2B.with_(n_layers=ecfg.n_layers, width=256, n_heads=4, head_dim=ecfg.head_dim, mlp_dim=512)
    w = make_llm_weights(cfg, 85, std=0.05)
    we = make_weights(ecfg, 86)
    B, P, C, N = 2, 40, 10, 3
    x = torch.from_numpy(make_prefix_embeddings(cfg, 87, B, P)).cuda()
    r = make_requests(ecfg, 88, B, 1, C)
    state, noise = torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda()
    pre = prefill.Prefill(cfg, w, max_batch=B, max_prefix=P)
    ex = make_expert(ecfg, we, max_batch=B, max_prefix=P, max_chunk=C, max_steps=N)
    pre.into_expert(x, ex, final=False)
    a = ex.denoise(state, noise, N)
    K, V, _ = pre.into_tensors(x, final=False)
    ex.set_prefix_kv(K, V)
    b = ex.denoise(state, noise, N)
    torch.cuda.synchronize()
    ex.device_status()
    pre.device_status()
    assert torch.equal(a, b)
    ex.close()
    pre.close()
