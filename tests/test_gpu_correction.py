"""Parity of the correction items (context tokens after the state token) on the CUDA path.

The correction module's predicted future VLM state (App. B, Alg. 1) reaches the expert as T'
context tokens; the oracle's reading R15 defines the result. Cases: the tiny fp32 expert
(CUDA-core path), the small bf16 expert over several tiles with both attention kernels, the
pi0.5-shaped expert at batch 1 (split-KV attention) and batch 8 (tcgen05 attention, large-M
gate/up), and the return to the plain expert when the items are cleared.
"""

import numpy as np
import pytest

import oracle
from synth import PI05, TINY, make_correction, make_requests, make_weights
from tests.gpu_util import SMALL_BF16, assert_close, errors, gpu_denoise, lib, make_expert, to_dev_kv

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    torch.cuda.set_device(0)
    lib()


def _oracle(cfg, w, r, corr, N, requests=None):
    req = list(range(r["noise"].shape[0])) if requests is None else list(requests)
    return oracle.denoise_batch(r["noise"][req], r["state"][req], N, r["prefix_k"][:, req],
                                r["prefix_v"][:, req], w, cfg, corr=corr[req])


def _set(ex, corr):
    ex.set_correction(torch.from_numpy(corr).cuda())


def test_tiny_fp32_forward_and_denoise_with_items():
    w = make_weights(TINY, 0)
    ex = make_expert(TINY, w, max_batch=2, max_prefix=64, max_chunk=8, max_steps=4)
    try:
        r = make_requests(TINY, 41, 2, 40, 6)
        corr = make_correction(TINY, 42, 2, 2)
        k, v = to_dev_kv(r, TINY)
        ex.set_prefix_kv(k, v)
        _set(ex, corr)
        vel, hres = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), 0.37)
        torch.cuda.synchronize()
        ref_v, ref_h = oracle.forward_batch(r["noise"], r["state"], 0.37, r["prefix_k"], r["prefix_v"], w,
                                            TINY, corr=corr)
        assert hres.shape == (2, 1 + 2 + 6, TINY.width)
        assert_close(vel.cpu().numpy(), ref_v, TINY, "tiny fp32 items forward v")
        assert np.abs(hres.cpu().numpy() - ref_h).max() <= 1e-4 * max(1.0, np.abs(ref_h).max())
        got = gpu_denoise(ex, TINY, r, 3)
        assert_close(got, _oracle(TINY, w, r, corr, 3), TINY, "tiny fp32 items denoise")
    finally:
        ex.close()


@pytest.mark.parametrize("attn", ["split_kv", "tcgen05"])
@pytest.mark.parametrize("B,P,C,T,N", [(2, 100, 13, 3, 2), (1, 257, 50, 4, 1), (3, 1, 1, 1, 2)])
def test_small_bf16_items(attn, B, P, C, T, N, monkeypatch):
    # Either attention kernel at every batch: 0 turns the tcgen05 kernel off, 1 takes it from one request.
    monkeypatch.setenv("JPI_ATTN_T5_MIN_BATCH", "1" if attn == "tcgen05" else "0")
    w = make_weights(SMALL_BF16, 2600, mod_bias_std=0.5)
    ex = make_expert(SMALL_BF16, w, max_batch=3, max_prefix=300, max_chunk=70, max_steps=3)
    try:
        r = make_requests(SMALL_BF16, 2601 + B, B, P, C)
        corr = make_correction(SMALL_BF16, 2602 + B, B, T, std=0.5)
        _set(ex, corr)
        got = gpu_denoise(ex, SMALL_BF16, r, N)
        assert_close(got, _oracle(SMALL_BF16, oracle.to_f64(w), r, corr, N), SMALL_BF16,
                     f"small bf16 items {attn} B{B} P{P} C{C} T{T} N{N}")
    finally:
        ex.close()


@pytest.fixture(scope="module")
def pi05():
    w = oracle.to_f64(make_weights(PI05, 2000))
    w32 = {k: v for k, v in w.items() if k != "__f64__"}
    ex = make_expert(PI05, w32, max_batch=8, max_prefix=816, max_chunk=50, max_steps=10)
    yield w, ex
    ex.close()


def test_pi05_batch1_four_items(pi05):
    w, ex = pi05
    r = make_requests(PI05, 2701, 1, 816, 50)
    corr = make_correction(PI05, 2702, 1, 4, std=0.5)
    _set(ex, corr)
    got = gpu_denoise(ex, PI05, r, 10)
    assert_close(got, _oracle(PI05, w, r, corr, 10), PI05, "pi0.5 items B1 P816 C50 T4 N10")


def test_pi05_batch8_four_items_sampled(pi05):
    w, ex = pi05
    r = make_requests(PI05, 2801, 8, 816, 50)
    corr = make_correction(PI05, 2802, 8, 4, std=0.5)
    _set(ex, corr)
    got = gpu_denoise(ex, PI05, r, 10)
    sample = [0, 7]
    assert_close(got[sample], _oracle(PI05, w, r, corr, 10, sample), PI05, "pi0.5 items B8 T4 sampled")


def test_pi05_items_change_the_actions_and_clearing_restores_the_plain_expert(pi05):
    w, ex = pi05
    r = make_requests(PI05, 2901, 1, 816, 50)
    ex.set_correction(None)
    plain = gpu_denoise(ex, PI05, r, 5)
    _set(ex, make_correction(PI05, 2902, 1, 4, std=0.5))
    with_items = gpu_denoise(ex, PI05, r, 5)
    ex.set_correction(None)
    again = gpu_denoise(ex, PI05, r, 5)
    np.testing.assert_array_equal(again, plain)          # same graph, same arithmetic
    assert errors(with_items, plain)[0] > 1e-3


def test_scheduler_drives_the_expert_with_predicted_states():
    """App. C Alg. 1 over the library: each chunk the scheduler stores is the expert's denoise
    for the state the (scripted) VLM or correction module produced, with the current KV."""
    from paper_2607_12659_gb300.scheduler import ConfidenceScheduler, expert_act
    w = make_weights(TINY, 0)
    ex = make_expert(TINY, w, max_batch=1, max_prefix=64, max_chunk=8, max_steps=4)
    try:
        r = make_requests(TINY, 51, 1, 40, 6)
        kv = to_dev_kv(r, TINY)
        h0 = torch.from_numpy(make_correction(TINY, 52, 1, 2)).cuda()
        h1 = torch.from_numpy(make_correction(TINY, 53, 1, 2)).cuda()
        state = torch.from_numpy(r["state"]).cuda()
        noise = torch.from_numpy(r["noise"]).cuda()
        act = expert_act(ex, lambda: state, lambda: noise, 3)
        sch = ConfidenceScheduler(vlm=lambda obs: (h0, kv), corr=lambda h, a: (h1, 0.5), act=act,
                                  observe=lambda: "obs", theta=-0.2, delta=4, delta_ae=2)
        sch.start()
        sch.iterate()                                # correction branch: predicted state h1
        torch.cuda.synchronize()
        ex.device_status()

        def direct(h):
            ex.set_prefix_kv(*kv)
            ex.set_correction(h)
            out = ex.denoise(state, noise, 3)
            torch.cuda.synchronize()
            return out.cpu().numpy()[0]

        first, second = direct(h0), direct(h1)
        got = sch.buffer.committed(2 + 6)
        np.testing.assert_array_equal(np.stack(got[:2]), first[:2])
        np.testing.assert_array_equal(np.stack(got[2:]), second)
        assert np.abs(first - second).max() > 1e-6
    finally:
        ex.close()
