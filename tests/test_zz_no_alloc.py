"""The allocation-free expert evaluation agrees with jpi_expert_forward.

jpi_expert_forward_noalloc serves callers that cannot call cudaMalloc: it keeps the scratch of
its time-conditioning stage in a fixed device array built into the library. Two calls in a row
(the second reuses the array the first left behind) must reproduce the velocity and hidden
state of jpi_expert_forward on the same inputs. This file runs last so that, if it fails, a run
that stops at the first failure has already run every other test.
"""

import numpy as np
import pytest

from synth import TINY, make_requests, make_weights
from tests.gpu_util import SMALL_BF16, FP32_MAX_ABS, BF16_MAX_ABS, lib, make_expert, to_dev_kv

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.mark.parametrize("cfg", [TINY, SMALL_BF16], ids=["fp32", "bf16"])
def test_noalloc_forward_matches_forward_twice(cfg):
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    torch.cuda.set_device(0)
    jpi = lib()
    w = make_weights(cfg, 41)
    ex = make_expert(cfg, w, max_batch=2, max_prefix=48, max_chunk=9, max_steps=2)
    try:
        r = make_requests(cfg, 42, 2, 48, 9)
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        s = torch.from_numpy(r["state"]).cuda()
        x = torch.from_numpy(r["noise"]).cuda()
        ref_v, ref_h = ex.forward(s, x, 0.45)
        torch.cuda.synchronize()
        ref_v, ref_h = ref_v.cpu().numpy(), ref_h.cpu().numpy()
        tol = FP32_MAX_ABS if cfg.precision == "fp32" else BF16_MAX_ABS
        for t, expect_v in ((0.45, ref_v), (0.45, ref_v)):
            out_v = torch.full_like(x, float("nan"))
            out_h = torch.full((2, 10, cfg.width), float("nan"), device="cuda")
            jpi.jpi_expert_forward_noalloc(ex.handle, s, x, t, 2, 9, out_v, out_h)
            torch.cuda.synchronize()
            ex.device_status()
            np.testing.assert_allclose(out_v.cpu().numpy(), expect_v, atol=tol, rtol=0)
            np.testing.assert_allclose(out_h.cpu().numpy(), ref_h, atol=tol * max(1.0, np.abs(ref_h).max()), rtol=0)
    finally:
        ex.close()
