"""The allocation-free expert evaluation agrees with jpi_expert_forward.

jpi_expert_forward_noalloc serves callers that cannot call cudaMalloc (code running inside a
stream capture, or under an allocator that owns all device memory): it keeps the scratch of
its time-conditioning stage in a fixed device array built into the library. Calls in a row at
different flow times (each one overwrites what the one before left in the array) must reproduce
the velocity and hidden state of jpi_expert_forward at the same t, and the oracle's velocity;
so must a call with correction items set, and a batch that differs from the items' batch is
refused as jpi_expert_forward refuses it. This file runs last so that, if it fails, a run that
stops at the first failure has already run every other test.
"""

import numpy as np
import pytest

import oracle
from synth import TINY, make_correction, make_requests, make_weights
from tests.gpu_util import (SMALL_BF16, FP32_MAX_ABS, BF16_MAX_ABS, assert_close, lib,
                            make_expert, to_dev_kv)

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

B, P, C = 2, 48, 9


def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    torch.cuda.set_device(0)


def _noalloc(jpi, ex, s, x, t, rows, width):
    out_v = torch.full_like(x, float("nan"))
    out_h = torch.full((B, rows, width), float("nan"), device="cuda")
    jpi.jpi_expert_forward_noalloc(ex.handle, s, x, t, B, C, out_v, out_h)
    torch.cuda.synchronize()
    ex.device_status()
    return out_v.cpu().numpy(), out_h.cpu().numpy()


def _check(cfg, w, r, ex, jpi, s, x, corr, what):
    tol = FP32_MAX_ABS if cfg.precision == "fp32" else BF16_MAX_ABS
    rows = 1 + (0 if corr is None else corr.shape[1]) + C
    # Two different flow times in turn: the second call must not see what the first left.
    for t in (0.9, 0.45):
        ref_v, ref_h = ex.forward(s, x, t)
        torch.cuda.synchronize()
        ref_v, ref_h = ref_v.cpu().numpy(), ref_h.cpu().numpy()
        got_v, got_h = _noalloc(jpi, ex, s, x, t, rows, cfg.width)
        np.testing.assert_allclose(got_v, ref_v, atol=tol, rtol=0, err_msg=f"{what} t={t}")
        np.testing.assert_allclose(got_h, ref_h, atol=tol * max(1.0, np.abs(ref_h).max()), rtol=0,
                                   err_msg=f"{what} t={t}")
        want_v, _ = oracle.forward_batch(r["noise"], r["state"], t, r["prefix_k"], r["prefix_v"], w,
                                         cfg, corr=corr)
        assert_close(got_v, want_v, cfg, f"noalloc {what} t={t} vs oracle")


@pytest.mark.parametrize("cfg", [TINY, SMALL_BF16], ids=["fp32", "bf16"])
def test_noalloc_forward_matches_forward_at_two_times(cfg):
    _cuda()
    jpi = lib()
    w = make_weights(cfg, 41)
    ex = make_expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=2)
    try:
        r = make_requests(cfg, 42, B, P, C)
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        s = torch.from_numpy(r["state"]).cuda()
        x = torch.from_numpy(r["noise"]).cuda()
        _check(cfg, w, r, ex, jpi, s, x, None, cfg.precision)
    finally:
        ex.close()


@pytest.mark.parametrize("cfg", [TINY, SMALL_BF16], ids=["fp32", "bf16"])
def test_noalloc_forward_with_correction_items(cfg):
    _cuda()
    jpi = lib()
    w = make_weights(cfg, 43)
    ex = make_expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=2)
    try:
        r = make_requests(cfg, 44, B, P, C)
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        corr = make_correction(cfg, 45, B, 3, std=0.5)
        ex.set_correction(torch.from_numpy(corr).cuda())
        s = torch.from_numpy(r["state"]).cuda()
        x = torch.from_numpy(r["noise"]).cuda()
        _check(cfg, w, r, ex, jpi, s, x, corr, f"{cfg.precision} items")
    finally:
        ex.close()


def test_noalloc_refuses_a_batch_other_than_the_items_batch():
    _cuda()
    jpi = lib()
    cfg = TINY
    w = make_weights(cfg, 46)
    ex = make_expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=2)
    try:
        r = make_requests(cfg, 47, B, P, C)
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        # Items for one request while the prefix holds two.
        ex.set_correction(torch.from_numpy(make_correction(cfg, 48, 1, 2)).cuda())
        s = torch.from_numpy(r["state"]).cuda()
        x = torch.from_numpy(r["noise"]).cuda()
        out_v = torch.empty_like(x)
        for call in (jpi.jpi_expert_forward, jpi.jpi_expert_forward_noalloc):
            with pytest.raises(jpi.JpiError) as e:
                call(ex.handle, s, x, 0.5, B, C, out_v)
            assert e.value.status == -2, (call.__name__, e.value)
        ex.device_status()
    finally:
        ex.close()
