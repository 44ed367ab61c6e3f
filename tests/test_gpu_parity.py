"""Parity of the CUDA path (through the C-ABI) with the fp64 CPU oracle on seeded inputs.

Configurations: the tiny fp32 expert; a small bf16 expert spanning several weight tiles with
ragged token counts; the pi0.5-shaped expert at batch 1 (816-token prefix, 50 x 32 chunk,
10 steps); its sweep over prefix length, chunk and step count; batches 4/8/16 with
per-request prefixes; and batch 64 with 2048-token prefixes (sampled requests).
"""

import numpy as np
import pytest

import oracle
from synth import PI05, TINY, ExpertConfig, make_requests, make_weights
from tests.gpu_util import (SMALL_BF16, assert_close, errors, gpu_denoise, lib, make_expert,
                            oracle_denoise, to_dev_kv)

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    torch.cuda.set_device(0)
    lib()


# ------------------------------------------------------------------ tiny fp32 (verification mode)

@pytest.fixture(scope="module")
def tiny():
    w = make_weights(TINY, 0)
    ex = make_expert(TINY, w, max_batch=3, max_prefix=64, max_chunk=8, max_steps=4)
    yield w, ex
    ex.close()


def test_tiny_fp32_denoise(tiny):
    w, ex = tiny
    r = make_requests(TINY, 1, 1, 64, 8)
    got = gpu_denoise(ex, TINY, r, 4)
    assert_close(got, oracle_denoise(TINY, w, r, 4), TINY, "tiny fp32")


@pytest.mark.parametrize("B,P,C,N", [(1, 1, 1, 1), (2, 63, 5, 3), (3, 17, 8, 2)])
def test_tiny_fp32_ragged_shapes(tiny, B, P, C, N):
    w, ex = tiny
    r = make_requests(TINY, 7, B, P, C)
    got = gpu_denoise(ex, TINY, r, N)
    assert_close(got, oracle_denoise(TINY, w, r, N), TINY, f"tiny fp32 B{B} P{P} C{C} N{N}")


def test_tiny_fp32_forward_velocity_and_hidden(tiny):
    w, ex = tiny
    r = make_requests(TINY, 3, 2, 40, 6)
    k, v = to_dev_kv(r, TINY)
    ex.set_prefix_kv(k, v)
    x = torch.from_numpy(r["noise"]).cuda()
    vel, hres = ex.forward(torch.from_numpy(r["state"]).cuda(), x, 0.37)
    torch.cuda.synchronize()
    ref_v, ref_h = oracle.forward_batch(r["noise"], r["state"], 0.37, r["prefix_k"], r["prefix_v"], w, TINY)
    assert_close(vel.cpu().numpy(), ref_v, TINY, "forward v")
    scale = np.abs(ref_h).max()
    assert np.abs(hres.cpu().numpy() - ref_h).max() <= 1e-4 * max(1.0, scale)


# ------------------------------------------------------------------ small bf16, several tiles

@pytest.fixture(scope="module")
def small():
    w = make_weights(SMALL_BF16, 11, mod_bias_std=0.5)
    ex = make_expert(SMALL_BF16, w, max_batch=5, max_prefix=300, max_chunk=70, max_steps=6)
    yield w, ex
    ex.close()


@pytest.mark.parametrize("B,P,C,N", [(1, 100, 13, 3), (2, 257, 50, 2), (5, 64, 70, 1), (3, 1, 1, 4)])
def test_small_bf16_denoise(small, B, P, C, N):
    w, ex = small
    r = make_requests(SMALL_BF16, 12, B, P, C)
    got = gpu_denoise(ex, SMALL_BF16, r, N)
    assert_close(got, oracle_denoise(SMALL_BF16, w, r, N), SMALL_BF16, f"small bf16 B{B} P{P} C{C} N{N}")


def test_small_bf16_forward_hidden_state(small):
    w, ex = small
    r = make_requests(SMALL_BF16, 13, 2, 150, 20)
    k, v = to_dev_kv(r, SMALL_BF16)
    ex.set_prefix_kv(k, v)
    vel, hres = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), 0.55)
    torch.cuda.synchronize()
    ref_v, ref_h = oracle.forward_batch(r["noise"], r["state"], 0.55, r["prefix_k"], r["prefix_v"], w, SMALL_BF16)
    assert_close(vel.cpu().numpy(), ref_v, SMALL_BF16, "small forward v")
    _, rel = errors(hres.cpu().numpy(), ref_h)
    assert rel <= 1e-2, f"hidden state rel-L2 {rel:.3g}"


# ------------------------------------------------------------------ pi0.5-shaped expert

@pytest.fixture(scope="module")
def pi05():
    w = oracle.to_f64(make_weights(PI05, 2000))
    w32 = {k: v for k, v in w.items() if k != "__f64__"}
    ex = make_expert(PI05, w32, max_batch=16, max_prefix=1536, max_chunk=50, max_steps=10)
    yield w, ex
    ex.close()


def test_pi05_batch1_prefix816_chunk50_steps10(pi05):
    w, ex = pi05
    r = make_requests(PI05, 2001, 1, 816, 50)
    got = gpu_denoise(ex, PI05, r, 10)
    max_abs, rel = assert_close(got, oracle_denoise(PI05, w, r, 10), PI05, "pi0.5 B1 P816 C50 N10")
    print(f"pi0.5 config: max-abs {max_abs:.3g} rel-L2 {rel:.3g}")


@pytest.mark.parametrize("P", [256, 512, 816, 1536])
@pytest.mark.parametrize("C", [10, 50])
@pytest.mark.parametrize("N", [1, 5, 10])
def test_pi05_sweep(pi05, P, C, N):
    w, ex = pi05
    r = make_requests(PI05, 3000 + P + C + N, 1, P, C)
    got = gpu_denoise(ex, PI05, r, N)
    assert_close(got, oracle_denoise(PI05, w, r, N), PI05, f"sweep P{P} C{C} N{N}")


@pytest.mark.parametrize("B", [4, 8, 16])
def test_pi05_batches_sampled_requests(pi05, B):
    w, ex = pi05
    r = make_requests(PI05, 4000 + B, B, 816, 50)
    got = gpu_denoise(ex, PI05, r, 10)
    sample = sorted({0, B // 2, B - 1})
    assert_close(got[sample], oracle_denoise(PI05, w, r, 10, sample), PI05, f"batch {B}")
    # Batch independence: request b alone gives the same actions as inside the batch, up to the
    # low-order bits that the attention's batch-dependent key split moves.
    b = B - 1
    r1 = make_requests(PI05, 4000 + B, 1, 816, 50, first_request=b)
    one = gpu_denoise(ex, PI05, r1, 10)
    assert_close(got[b:b + 1], one, PI05, f"batch {B} vs alone")


def test_pi05_high_gain_forward():
    """Gates of O(1) (modulation biases ~N(0,1)) so every sublayer visibly moves the output."""
    w = make_weights(PI05.with_(n_layers=4), 2100, mod_bias_std=1.0)
    cfg = PI05.with_(n_layers=4)
    ex = make_expert(cfg, w, max_batch=2, max_prefix=816, max_chunk=50, max_steps=1)
    try:
        r = make_requests(cfg, 2101, 2, 816, 50)
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        vel, hres = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), 0.3)
        torch.cuda.synchronize()
        ref_v, ref_h = oracle.forward_batch(r["noise"], r["state"], 0.3, r["prefix_k"], r["prefix_v"], w, cfg)
        # Stress variant, not one of the five workloads: O(1) gates amplify the bf16 rounding
        # of every tensor-core input, so max-abs gets 3e-2; rel-L2 keeps the 1e-2 contract.
        assert_close(vel.cpu().numpy(), ref_v, cfg, "high-gain forward v", max_abs_tol=3e-2)
        _, rel = errors(hres.cpu().numpy(), ref_h)
        assert rel <= 1e-2, f"high-gain hidden rel-L2 {rel:.3g}"
    finally:
        ex.close()


def test_pi05_batch64_prefix2048_sampled():
    w = make_weights(PI05, 2000)
    ex = make_expert(PI05, w, max_batch=64, max_prefix=2048, max_chunk=50, max_steps=10)
    try:
        r = make_requests(PI05, 5000, 64, 2048, 50)
        got = gpu_denoise(ex, PI05, r, 10)
        sample = [0, 21, 42, 63]
        assert_close(got[sample], oracle_denoise(PI05, w, r, 10, sample), PI05, "batch 64 P2048")
    finally:
        ex.close()


@pytest.fixture
def large_m_everywhere(monkeypatch):
    """Handles created under this fixture run every projection through the large-M kernel."""
    monkeypatch.setenv("JPI_BIG_GEMM_MIN_TOKENS", "1")


@pytest.mark.parametrize("B,P,C,N", [(1, 100, 13, 2), (3, 257, 50, 1), (2, 64, 70, 3)])
def test_small_bf16_large_m_projection_path(large_m_everywhere, B, P, C, N):
    w = make_weights(SMALL_BF16, 2200)
    ex = make_expert(SMALL_BF16, w, max_batch=3, max_prefix=300, max_chunk=70, max_steps=3)
    try:
        r = make_requests(SMALL_BF16, 2201 + B, B, P, C)
        got = gpu_denoise(ex, SMALL_BF16, r, N)
        assert_close(got, oracle_denoise(SMALL_BF16, oracle.to_f64(w), r, N), SMALL_BF16,
                     f"small bf16 large-M B{B} P{P} C{C} N{N}")
    finally:
        ex.close()


# One head of 128: the QKV projection has an odd number of weight tiles (3), and a single
# 128-row weight tile carries both halves of the head's rotary pairs.
SMALL_ONE_HEAD = ExpertConfig(n_layers=2, width=256, n_heads=1, head_dim=128, mlp_dim=512,
                              action_dim=7, state_dim=7, time_dim=64, precision="bf16")


@pytest.mark.parametrize("B,P,C", [(2, 100, 50), (5, 64, 31)])
def test_odd_weight_tile_count_large_m_path(large_m_everywhere, B, P, C):
    w = make_weights(SMALL_ONE_HEAD, 2250)
    ex = make_expert(SMALL_ONE_HEAD, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=2)
    try:
        r = make_requests(SMALL_ONE_HEAD, 2251 + B, B, P, C)
        got = gpu_denoise(ex, SMALL_ONE_HEAD, r, 2)
        assert_close(got, oracle_denoise(SMALL_ONE_HEAD, oracle.to_f64(w), r, 2), SMALL_ONE_HEAD,
                     f"one-head large-M B{B} P{P} C{C}")
    finally:
        ex.close()


# The large-M residual projections (O, down) may split each unit's K range over a cluster of
# 1, 2, 4 or 8 CTAs, exchanging fp32 partials and summing them in rank order (JPI_BIG_SPLIT fixes
# the split). Every split must match the oracle; between splits only the order of the fp32 sums
# of the partials differs, which can move a bf16 rounding of the next projection's operand (2^-9
# relative), so two layers' hidden states must agree to 2e-3 of their largest magnitude.
BIG_SPLITS = (1, 2, 4, 8)


def test_pi05_large_m_k_splits(large_m_everywhere, monkeypatch):
    cfg = PI05.with_(n_layers=2)
    w = make_weights(cfg, 2280)
    r = make_requests(cfg, 2281, 4, 816, 50)
    t = 0.6
    want_v, want_h = oracle.forward_batch(r["noise"], r["state"], t, r["prefix_k"], r["prefix_v"], w, cfg)
    got = {}
    for S in BIG_SPLITS:
        monkeypatch.setenv("JPI_BIG_SPLIT", str(S))
        ex = make_expert(cfg, w, max_batch=4, max_prefix=816, max_chunk=50, max_steps=1)
        try:
            k, v = to_dev_kv(r, cfg)
            ex.set_prefix_kv(k, v)
            vel, hid = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), t)
            torch.cuda.synchronize()
            ex.device_status()
            got[S] = (vel.cpu().numpy(), hid.cpu().numpy())
        finally:
            ex.close()
        assert_close(got[S][0], want_v, cfg, f"pi0.5 2 layers B4, large-M K split {S}")
        _, rel = errors(got[S][1], want_h)
        assert rel <= 1e-2, f"K split {S}: hidden rel-L2 {rel:.3g}"
    scale = float(np.abs(want_h).max())
    for S in BIG_SPLITS[1:]:
        dh = float(np.abs(got[S][1] - got[1][1]).max()) / scale
        print(f"K split {S} vs 1: hidden {dh:.3g} of max |h|")
        assert dh <= 2e-3, f"K split {S} vs 1: hidden state differs by {dh:.3g} of max |h|"


def test_pi05_large_m_projection_path(large_m_everywhere):
    w = make_weights(PI05, 2000)
    ex = make_expert(PI05, w, max_batch=3, max_prefix=816, max_chunk=50, max_steps=10)
    try:
        r = make_requests(PI05, 2300, 3, 816, 50)
        got = gpu_denoise(ex, PI05, r, 10)
        assert_close(got[[0, 2]], oracle_denoise(PI05, w, r, 10, [0, 2]), PI05, "pi0.5 large-M B3")
    finally:
        ex.close()


@pytest.fixture
def tcgen05_attention_everywhere(monkeypatch):
    """Handles created under this fixture take the tcgen05 attention at any batch (its keys split
    four ways where the clusters fit, as chosen per launch)."""
    monkeypatch.setenv("JPI_ATTN_T5_MIN_BATCH", "1")


@pytest.mark.parametrize("B,P,C,N", [(1, 100, 13, 2), (3, 257, 50, 1), (2, 64, 70, 3), (1, 1, 1, 2)])
def test_small_bf16_tcgen05_attention(tcgen05_attention_everywhere, B, P, C, N):
    w = make_weights(SMALL_BF16, 2400)
    ex = make_expert(SMALL_BF16, w, max_batch=3, max_prefix=300, max_chunk=70, max_steps=3)
    try:
        r = make_requests(SMALL_BF16, 2401 + B, B, P, C)
        got = gpu_denoise(ex, SMALL_BF16, r, N)
        assert_close(got, oracle_denoise(SMALL_BF16, oracle.to_f64(w), r, N), SMALL_BF16,
                     f"small bf16 tcgen05 attention B{B} P{P} C{C} N{N}")
    finally:
        ex.close()


def test_small_bf16_tcgen05_attention_rescales(tcgen05_attention_everywhere):
    """O(1) modulation gains give score spreads wide enough that the running maximum moves by
    more than the lazy-rescale threshold inside a row."""
    w = make_weights(SMALL_BF16, 2410, mod_bias_std=1.0)
    ex = make_expert(SMALL_BF16, w, max_batch=2, max_prefix=300, max_chunk=70, max_steps=2)
    try:
        r = make_requests(SMALL_BF16, 2411, 2, 300, 70)
        got = gpu_denoise(ex, SMALL_BF16, r, 2)
        assert_close(got, oracle_denoise(SMALL_BF16, oracle.to_f64(w), r, 2), SMALL_BF16,
                     "small bf16 tcgen05 attention high gain", max_abs_tol=3e-2)
    finally:
        ex.close()


def test_pi05_tcgen05_attention(tcgen05_attention_everywhere):
    w = make_weights(PI05, 2000)
    ex = make_expert(PI05, w, max_batch=2, max_prefix=1536, max_chunk=50, max_steps=10)
    try:
        for P in (816, 1536):
            r = make_requests(PI05, 2500 + P, 2, P, 50)
            got = gpu_denoise(ex, PI05, r, 10)
            assert_close(got[[1]], oracle_denoise(PI05, w, r, 10, [1]), PI05, f"pi0.5 tcgen05 attention B2 P{P}")
    finally:
        ex.close()


# Split-KV combine: the attention's result does not depend on how many key splits it was
# computed in (JPI_ATTN_SPLITS fixes the count at create time; 16 asks for the largest cluster,
# 14 splits of 64 keys at 867 keys). On the full expert every split count must match the oracle.
# Between split counts the only differences are roundings: each split's unnormalised output is
# rounded to fp16 (2^-11 relative) before the combine, the fp32 sums run in another order, and
# the combined output is rounded to bf16 (2^-9). One layer carries them to its output without the
# 18-layer growth, so there the split counts must agree to SPLIT_AGREEMENT (relative to the
# largest output magnitude).
SPLIT_COUNTS = (1, 2, 7, 16)
SPLIT_AGREEMENT = 2e-3


def _forward_with_splits(monkeypatch, cfg, w, r, t, splits):
    monkeypatch.setenv("JPI_ATTN_SPLITS", str(splits))
    P, C = r["prefix_k"].shape[2], r["noise"].shape[1]
    ex = make_expert(cfg, w, max_batch=1, max_prefix=P, max_chunk=C, max_steps=1)
    try:
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        vel, hid = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), t)
        torch.cuda.synchronize()
        ex.device_status()
        return vel.cpu().numpy(), hid.cpu().numpy()
    finally:
        ex.close()


def test_pi05_every_split_count_matches_the_oracle(monkeypatch):
    w = make_weights(PI05, 2000)
    r = make_requests(PI05, 2600, 1, 816, 50)
    t = 0.3
    want, _ = oracle.forward_batch(r["noise"], r["state"], t, r["prefix_k"], r["prefix_v"], w, PI05)
    for splits in SPLIT_COUNTS:
        vel, _ = _forward_with_splits(monkeypatch, PI05, w, r, t, splits)
        assert_close(vel, want, PI05, f"pi0.5 forward P816, {splits} key splits")


def test_split_counts_agree_on_one_pi05_shaped_layer(monkeypatch):
    cfg = PI05.with_(n_layers=1)
    w = make_weights(cfg, 2610)
    r = make_requests(cfg, 2611, 1, 816, 50)
    t = 0.3
    want_v, want_h = oracle.forward_batch(r["noise"], r["state"], t, r["prefix_k"], r["prefix_v"], w, cfg)
    got = {s: _forward_with_splits(monkeypatch, cfg, w, r, t, s) for s in SPLIT_COUNTS}
    scale = float(np.abs(want_h).max())
    for s in SPLIT_COUNTS:
        assert_close(got[s][0], want_v, cfg, f"one pi0.5 layer, {s} key splits")
    for s in SPLIT_COUNTS[:-1]:
        dh = float(np.abs(got[s][1] - got[16][1]).max()) / scale
        dv = float(np.abs(got[s][0] - got[16][0]).max())
        print(f"splits {s} vs 14: hidden {dh:.3g} (relative to max |h| {scale:.3g}), velocity {dv:.3g}")
        assert dh <= SPLIT_AGREEMENT, f"{s} key splits: hidden state differs by {dh:.3g} of max |h|"


# The tcgen05 attention's key split: the key blocks of each 128-row block spread over a cluster of
# 1-4 CTAs whose fp32 partial rows are combined in split order through a workspace in global
# memory (JPI_ATTN_T5_SPLITS fixes the count; 2 and 4 keep each CTA's own rows on chip, 3 takes
# the general combine). Every count must match the oracle; between counts only the fp32 rounding
# of the combine differs.
T5_SPLITS = (1, 2, 3, 4)


def _forward_t5_splits(monkeypatch, cfg, w, r, t, splits):
    monkeypatch.setenv("JPI_ATTN_T5_MIN_BATCH", "1")
    monkeypatch.setenv("JPI_ATTN_T5_SPLITS", str(splits))
    B, P, C = r["noise"].shape[0], r["prefix_k"].shape[2], r["noise"].shape[1]
    ex = make_expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=1)
    try:
        k, v = to_dev_kv(r, cfg)
        ex.set_prefix_kv(k, v)
        vel, hid = ex.forward(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), t)
        torch.cuda.synchronize()
        ex.device_status()
        return vel.cpu().numpy(), hid.cpu().numpy()
    finally:
        ex.close()


def test_tcgen05_attention_key_splits_on_one_pi05_layer(monkeypatch):
    cfg = PI05.with_(n_layers=1)
    w = make_weights(cfg, 2620)
    r = make_requests(cfg, 2621, 2, 816, 50)
    t = 0.4
    want_v, want_h = oracle.forward_batch(r["noise"], r["state"], t, r["prefix_k"], r["prefix_v"], w, cfg)
    got = {s: _forward_t5_splits(monkeypatch, cfg, w, r, t, s) for s in T5_SPLITS}
    scale = float(np.abs(want_h).max())
    for s in T5_SPLITS:
        assert_close(got[s][0], want_v, cfg, f"one pi0.5 layer B2, tcgen05 attention, {s} key splits")
    for s in T5_SPLITS[1:]:
        dh = float(np.abs(got[s][1] - got[1][1]).max()) / scale
        print(f"tcgen05 attention {s} splits vs 1: hidden {dh:.3g} of max |h|")
        assert dh <= SPLIT_AGREEMENT, f"{s} key splits: hidden state differs by {dh:.3g} of max |h|"


@pytest.mark.parametrize("splits", [2, 4])
def test_tcgen05_attention_key_splits_small_and_ragged(monkeypatch, splits):
    # Prefix 70 + suffix 14 = 84 keys: two 64-key blocks, so 4 splits are capped at 2; the state
    # row sees the prefix and itself only.
    w = make_weights(SMALL_BF16, 2630)
    r = make_requests(SMALL_BF16, 2631, 3, 70, 13)
    t = 0.8
    want_v, _ = oracle.forward_batch(r["noise"], r["state"], t, r["prefix_k"], r["prefix_v"],
                                     oracle.to_f64(w), SMALL_BF16)
    vel, _ = _forward_t5_splits(monkeypatch, SMALL_BF16, w, r, t, splits)
    assert_close(vel, want_v, SMALL_BF16, f"small bf16 B3 P70, tcgen05 attention, {splits} key splits")


# Batch invariance, bit for bit: with JPI_BATCH_INVARIANT=1 every launch makes the choices it makes
# for a single request (the K-split projections with their fixed K split, the split-KV attention
# with one request's key split), so request b of a batch gets exactly the actions it gets alone.
# Without the switch the attention's split and the projection kernel follow the batch size and the
# low-order bits may move (test_pi05_batches_sampled_requests bounds that).
@pytest.mark.parametrize("cfg,P,C,N,B", [(SMALL_BF16, 100, 13, 2, 3), (PI05, 816, 50, 10, 16)],
                         ids=["small-bf16", "pi05"])
def test_batch_invariant_mode_is_bitwise(monkeypatch, cfg, P, C, N, B):
    monkeypatch.setenv("JPI_BATCH_INVARIANT", "1")
    w = make_weights(cfg, 2800)
    ex = make_expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=N)
    try:
        r = make_requests(cfg, 2801, B, P, C)
        got = gpu_denoise(ex, cfg, r, N)
        for b in sorted({0, B // 2, B - 1}):
            one = gpu_denoise(ex, cfg, make_requests(cfg, 2801, 1, P, C, first_request=b), N)
            assert np.array_equal(got[b:b + 1], one), \
                f"request {b}: max difference {float(np.abs(got[b:b + 1] - one).max()):.3g}"
        sample = [0, B - 1]
        assert_close(got[sample], oracle_denoise(cfg, oracle.to_f64(w), r, N, sample), cfg,
                     f"batch-invariant mode B{B} P{P}")
    finally:
        ex.close()
