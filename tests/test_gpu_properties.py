"""Properties of the CUDA path that hold at any size: closed forms, one step = one forward,
determinism, graph reuse across prefixes, host/device entry points, zero-copy KV, errors."""

import numpy as np
import pytest

from synth import TINY, make_requests, make_weights
from tests.gpu_util import SMALL_BF16, gpu_denoise, lib, make_expert, to_dev_kv

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

CONFIGS = [TINY, SMALL_BF16]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    torch.cuda.set_device(0)
    lib()


@pytest.mark.parametrize("cfg", CONFIGS, ids=["fp32", "bf16"])
@pytest.mark.parametrize("N", [1, 4, 7])
def test_zero_velocity_head_integrates_to_noise_plus_bias(cfg, N):
    w = make_weights(cfg, 21)
    c = np.linspace(-1.0, 1.0, cfg.action_dim).astype(np.float32)
    w["action_out_w"] = np.zeros_like(w["action_out_w"])
    w["action_out_b"] = c
    ex = make_expert(cfg, w, max_batch=2, max_prefix=40, max_chunk=9, max_steps=8)
    try:
        r = make_requests(cfg, 22, 2, 40, 9)
        got = gpu_denoise(ex, cfg, r, N)
        np.testing.assert_allclose(got, r["noise"] + c, atol=2e-6 * N, rtol=0)
    finally:
        ex.close()


@pytest.mark.parametrize("cfg", CONFIGS, ids=["fp32", "bf16"])
def test_one_step_equals_noise_plus_forward_at_t0(cfg):
    w = make_weights(cfg, 23)
    ex = make_expert(cfg, w, max_batch=2, max_prefix=50, max_chunk=8, max_steps=2)
    try:
        r = make_requests(cfg, 24, 2, 50, 8)
        one = gpu_denoise(ex, cfg, r, 1)
        v, _ = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), 0.0)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(one, r["noise"] + v.cpu().numpy())
    finally:
        ex.close()


@pytest.mark.parametrize("cfg", CONFIGS, ids=["fp32", "bf16"])
def test_bitwise_determinism_across_replays_and_handles(cfg):
    w = make_weights(cfg, 25)
    r = make_requests(cfg, 26, 2, 33, 7)
    outs = []
    for _ in range(2):
        ex = make_expert(cfg, w, max_batch=2, max_prefix=40, max_chunk=8, max_steps=5)
        try:
            for _ in range(3):
                outs.append(gpu_denoise(ex, cfg, r, 5))
        finally:
            ex.close()
    for o in outs[1:]:
        np.testing.assert_array_equal(o, outs[0])


def test_graph_cache_survives_prefix_changes():
    cfg = SMALL_BF16
    w = make_weights(cfg, 27)
    ex = make_expert(cfg, w, max_batch=1, max_prefix=200, max_chunk=10, max_steps=3)
    try:
        r1 = make_requests(cfg, 28, 1, 100, 10)
        r2 = make_requests(cfg, 29, 1, 180, 10)
        a = gpu_denoise(ex, cfg, r1, 3)
        b = gpu_denoise(ex, cfg, r2, 3)
        a2 = gpu_denoise(ex, cfg, r1, 3)
        np.testing.assert_array_equal(a, a2)
        assert np.abs(a - b).max() > 0
    finally:
        ex.close()


def test_host_entry_point_matches_device_entry_point():
    cfg = SMALL_BF16
    w = make_weights(cfg, 30)
    ex = make_expert(cfg, w, max_batch=2, max_prefix=64, max_chunk=12, max_steps=4)
    try:
        r = make_requests(cfg, 31, 2, 64, 12)
        dev = gpu_denoise(ex, cfg, r, 4)
        host = ex.denoise_host(r["state"], r["noise"], 4)
        np.testing.assert_array_equal(host, dev)
    finally:
        ex.close()


class _DeviceArray:
    """A raw device pointer exposed through __cuda_array_interface__ (so torch can view it)."""

    def __init__(self, ptr, shape, typestr):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (int(ptr), False), "version": 2, "strides": None}


def test_zero_copy_prefix_store_matches_copy_in():
    cfg = SMALL_BF16
    jpi = lib()
    w = make_weights(cfg, 32)
    ex = make_expert(cfg, w, max_batch=2, max_prefix=64, max_chunk=6, max_steps=2)
    try:
        B, P, C = 2, 50, 6
        r = make_requests(cfg, 33, B, P, C)
        ref = gpu_denoise(ex, cfg, r, 2)
        k, v = to_dev_kv(r, cfg)
        # Clear the store through the same pointers first, so the test sees the producer's writes.
        for l in range(cfg.n_layers):
            kp, vp, stride = jpi.jpi_prefix_kv_ptr(ex.handle, l)
            for b in range(B):
                for src, base in ((k[l, b], kp), (v[l, b], vp)):
                    dst = torch.as_tensor(_DeviceArray(base + 2 * b * stride, src.shape, "<i2"),
                                          device="cuda")
                    dst.zero_()
                    dst.copy_(src.view(torch.int16))
        jpi.jpi_commit_prefix(ex.handle, B, P)
        out = ex.denoise(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), 2)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(out.cpu().numpy(), ref)
    finally:
        ex.close()


def test_errors_are_status_codes():
    cfg = SMALL_BF16
    jpi = lib()
    w = make_weights(cfg, 34)
    ex = make_expert(cfg, w, max_batch=2, max_prefix=32, max_chunk=4, max_steps=2)
    try:
        s = torch.zeros(2, cfg.state_dim, device="cuda")
        x = torch.zeros(2, 4, cfg.action_dim, device="cuda")
        with pytest.raises(jpi.JpiError) as e:
            jpi.jpi_denoise(ex.handle, s, x, 2, 4, 2, x)
        assert e.value.status == -5                              # NOT_READY
        r = make_requests(cfg, 35, 2, 32, 4)
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        for args, status in [((2, 4, 3), -2), ((2, 5, 2), -2), ((2, 4, 0), -1), ((1, 4, 2), -2),
                             ((3, 4, 2), -2), ((0, 4, 2), -1)]:
            with pytest.raises(jpi.JpiError) as e:
                jpi.jpi_denoise(ex.handle, s, x, *args, x)
            assert e.value.status == status, (args, e.value)
        with pytest.raises(jpi.JpiError) as e:
            jpi.jpi_denoise(ex.handle, None, x, 2, 4, 2, x)
        assert e.value.status == -1
        with pytest.raises(jpi.JpiError) as e:
            jpi.jpi_set_prefix_kv(ex.handle, [k[l] for l in range(cfg.n_layers)],
                                  [v[l] for l in range(cfg.n_layers)], 2, 33, False)
        assert e.value.status == -2
        # The handle still works after the rejected calls.
        assert np.isfinite(gpu_denoise(ex, cfg, r, 2)).all()
    finally:
        ex.close()


def test_out_of_memory_is_a_status_and_frees_everything():
    # Maxima the shape checks accept but whose KV store cannot fit (about 56 TB): create fails with
    # JPI_ERR_OOM after about 14 GB of other buffers, and gives every one of them back.
    jpi = lib()
    cfg = TINY
    w = make_weights(cfg, 36)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    with pytest.raises(jpi.JpiError) as e:
        jpi.Expert(cfg, w, max_batch=(1 << 20) // 10, max_prefix=1 << 20, max_chunk=1, max_steps=1)
    assert e.value.status == -3, e.value
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert abs(free1 - free0) < (64 << 20)
