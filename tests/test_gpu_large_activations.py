"""Large activations through the partial exchanges of the CUDA path.

The split-K projections and the split-KV attention hand their partial results between the CTAs
of a cluster as fp16 (range 65504, 11 significant bits) before summing them in fp32; a value out
of that range stops the call with a device error instead of overflowing. These cases drive the
path at Gemma-like scales: prefix values V scaled by 128 or 512 (exact in bf16, so std 128 or 512 instead of 1)
and every attention and MLP gate shifted by +30, which grows the residual stream to 1e3..1e4
while the final adaptive norm keeps the velocity O(1). They must meet the oracle at the parity
tolerance with no device error, and the residual stream must really reach that scale.
"""

import numpy as np
import pytest

import oracle
from synth import PI05, make_requests, make_weights
from tests.gpu_util import SMALL_BF16, assert_close, gpu_denoise, lib, make_expert, oracle_denoise, to_dev_kv

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

GATE_SHIFT = 30.0


def _large(cfg, w, r, v_scale):
    """Gates (rows 2W..3W of both modulation biases) shifted by +30, prefix V times v_scale (a
    power of two, so the bf16 values stay exact)."""
    W = cfg.width
    w = dict(w)
    for name in ("attn_mod_b", "mlp_mod_b"):
        layers = []
        for b in w[name]:
            b = b.copy()
            b[2 * W:] += np.float32(GATE_SHIFT)
            layers.append(b)
        w[name] = layers
    r = dict(r)
    r["prefix_v"] = (r["prefix_v"] * np.float32(v_scale)).astype(np.float32)
    return w, r


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    torch.cuda.set_device(0)
    lib()


# Two layers need larger values than eighteen to reach the same residual scale.
@pytest.mark.parametrize("cfg,B,P,C,N,v_scale", [(SMALL_BF16, 2, 100, 13, 2, 512.0), (PI05, 1, 816, 50, 10, 128.0)],
                         ids=["small-bf16", "pi05-b1"])
def test_large_residual_stream_and_values(cfg, B, P, C, N, v_scale):
    w, r = _large(cfg, make_weights(cfg, 2700), make_requests(cfg, 2701, B, P, C), v_scale)
    ex = make_expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=N)
    try:
        # The scale the residual stream reaches (first Euler step, t = 0).
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        _, hid = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), 0.0)
        torch.cuda.synchronize()
        ex.device_status()
        peak = float(hid.abs().max())
        _, want_h = oracle.forward_batch(r["noise"], r["state"], 0.0, r["prefix_k"], r["prefix_v"], w, cfg)
        assert 1e3 <= float(np.abs(want_h).max()) and 1e3 <= peak, peak
        # The whole denoise, against the oracle (device errors, fp16 range included, raise).
        got = gpu_denoise(ex, cfg, r, N)
        assert_close(got, oracle_denoise(cfg, oracle.to_f64(w), r, N), cfg,
                     f"large activations {cfg.n_layers} layers B{B} P{P} (max |h| {peak:.3g})")
    finally:
        ex.close()
