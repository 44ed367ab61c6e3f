"""Host logic of bench.py: the roofline byte and FLOP counts against an independent count from
the weight shapes, the per-launch byte split, the clock-record parsing and the JSON contract of
the reference arm. No GPU is used."""

import json
import os
import subprocess
import sys

import numpy as np
import pytest

import bench
from synth import PI05, TINY, weight_shapes

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LAYER_PROJ = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")


def _size(shape):
    return int(np.prod(shape))


@pytest.mark.parametrize("cfg", [PI05, TINY], ids=["pi05", "tiny"])
@pytest.mark.parametrize("B,P,C,N", [(1, 816, 50, 10), (4, 300, 10, 3)])
def test_algorithmic_bytes_from_the_weight_shapes(cfg, B, P, C, N):
    ws = weight_shapes(cfg)
    L = cfg.n_layers
    step = 2 * (L * sum(_size(ws[k]) for k in LAYER_PROJ)
                + _size(ws["state_in_w"]) + _size(ws["action_in_w"]) + _size(ws["action_out_w"]))
    time_w = 2 * (_size(ws["time_mlp_in_w"]) + _size(ws["time_mlp_out_w"])
                  + L * (_size(ws["attn_mod_w"]) + _size(ws["mlp_mod_w"])) + _size(ws["final_mod_w"]))
    kv = B * L * P * cfg.head_dim * 2 * 2
    io = B * (cfg.state_dim + 2 * C * cfg.action_dim) * 4
    assert bench.algorithmic_bytes(cfg, B, P, C, N) == N * step + time_w + kv + io


def test_pi05_step_weights_are_the_paper_sized_expert():
    # 18 layers x 17,301,504 projection parameters + in/out projections, bf16: 623.05 MB.
    ws = weight_shapes(PI05)
    assert sum(_size(ws[k]) for k in LAYER_PROJ) == 17_301_504
    assert bench.algorithmic_bytes(PI05, 1, 816, 50, 10) == 6_480_441_984


@pytest.mark.parametrize("B,P,C,N,T", [(1, 816, 50, 10, 0), (64, 2048, 50, 10, 0), (3, 17, 8, 2, 0),
                                       (1, 816, 50, 10, 4)])
def test_algorithmic_flops_from_the_weight_shapes(B, P, C, N, T):
    cfg = PI05
    ws = weight_shapes(cfg)
    L, H, D, W = cfg.n_layers, cfg.n_heads, cfg.head_dim, cfg.width
    S = C + 1 + T                                  # state token, T correction items, C actions
    macs_step = (B * S * L * sum(_size(ws[k]) for k in LAYER_PROJ)
                 + L * B * 2 * (S * H) * (P + S) * D                       # QK^T and PV
                 + B * _size(ws["state_in_w"]) + B * C * _size(ws["action_in_w"])
                 + B * C * _size(ws["action_out_w"]))
    macs_time = (_size(ws["time_mlp_in_w"]) + _size(ws["time_mlp_out_w"])
                 + L * (_size(ws["attn_mod_w"]) + _size(ws["mlp_mod_w"])) + _size(ws["final_mod_w"]))
    assert bench.algorithmic_flops(cfg, B, P, C, N, T) == 2 * N * (macs_step + macs_time)


def test_layer_op_bytes_cover_each_layer_weight_once():
    cfg, B, P, C = PI05, 2, 816, 50
    ws = weight_shapes(cfg)
    Mt = B * (C + 1)
    W, F, HD, D = cfg.width, cfg.mlp_dim, cfg.n_heads * cfg.head_dim, cfg.head_dim
    acts = {2: Mt * W * 4 + Mt * (HD + 2 * D) * 2,       # h in, q/k/v out
            3: B * (P + C + 1) * D * 2 * 2 + Mt * HD * 2 * 2,
            4: Mt * HD * 2 + Mt * W * 4 * 2,
            5: Mt * W * 4 + Mt * F * 2,
            6: Mt * F * 2 + Mt * W * 4 * 2}
    weights = sum(bench.op_bytes(cfg, op, B, P, C) - acts[op] for op in range(2, 7))
    assert weights == 2 * sum(_size(ws[k]) for k in LAYER_PROJ)
    assert bench.op_bytes(cfg, 3, B, P, C) == acts[3]           # attention reads no weights


def test_clock_record_parsing():
    c = bench.ClockSampler(0)
    c.lines = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
               "0, 1980, 2070, 1399.0, 0x4, Not Active, Not Active, Not Active, Active",
               "0, 2070, 2070, 1200.0, 0x0, Not Active, Not Active, Not Active, Not Active",
               "garbage line"]
    s = c.summary()
    assert s == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    c.lines = []
    assert c.summary()["reasons"] == ["unavailable"]


def test_reference_arm_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "3"], capture_output=True, text=True, timeout=600,
                         cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0


def test_every_kernel_source_is_accounted_for_by_the_source_hash():
    # Every source of the expert's kernels changes `source_sha`, the build's identity in the bench
    # line; only the correction module's files stay outside.
    d = os.path.join(bench.ROOT, "paper_2607_12659_gb300", "csrc")
    files = {f for f in os.listdir(d) if f.endswith((".cu", ".cuh", ".h"))}
    assert files == set(bench.EXPERT_SOURCES) | set(bench.CORRECTION_SOURCES)
    assert not set(bench.EXPERT_SOURCES) & set(bench.CORRECTION_SOURCES)


def _local_include_closure(d, roots):
    seen, todo = set(), list(roots)
    while todo:
        f = todo.pop()
        if f in seen or not os.path.exists(os.path.join(d, f)):
            continue   # headers outside the kernel directory (the public ABI header) are not hashed
        seen.add(f)
        for line in open(os.path.join(d, f)):
            line = line.strip()
            if line.startswith('#include "'):
                todo.append(line.split('"')[1])
    return seen


def test_traffic_hash_covers_the_batch1_layer_kernels_and_their_headers():
    # The recorded DRAM traffic of the five batch-1 layer kernels (the projection kernel in
    # gemm_kernel.cuh, launched from tc_path.cu, and the split-KV attention in attn_tc.cu) stays
    # valid exactly while these files and every local header they include are unchanged.
    d = os.path.join(bench.ROOT, "paper_2607_12659_gb300", "csrc")
    closure = _local_include_closure(d, ["tc_path.cu", "attn_tc.cu"])
    assert closure == set(bench.TRAFFIC_SOURCES)
    assert set(bench.TRAFFIC_SOURCES) <= set(bench.EXPERT_SOURCES)
    for entry in bench.NCU_TRAFFIC.values():
        assert len(entry["source_sha256"]) == 16 and entry["bytes"] > 0


def test_correction_bytes_from_the_weight_shapes():
    # Per-call weights: everything but the compressor's query-side tensors, which create time
    # folds into the queries mapped into VLM space; plus the bf16 VLM output and the small I/O.
    from synth.correction import PI05_CORRECTION as c
    d, F, dv, A = c.width, c.mlp_dim, c.d_vlm, c.action_dim
    block_mats = 4 * d * d + 2 * d * F
    block_vecs = 4 * d + 4 * d + F + d           # ln1, ln2 (w, b), q/k/v/o biases, b1, b2
    mats = (d * dv + d * d + 2 * d * F          # compressor: value, output, MLP
            + d * A + d * d + c.max_delta * d    # action MLP, position table
            + block_mats * (1 + c.n_joint) + 2 * d * d + d * d + d)   # blocks, fuse, corr, conf
    vecs = (3 * d + F + 2 * d + 2 * d            # compressor: b_v, b_o, b2; b1; ln3; lnf
            + 2 * d                              # action biases
            + block_vecs * (1 + c.n_joint) + d + 2 * d + d + 1)   # fuse b, head ln, corr b, conf b
    want_w = 2 * (mats - c.max_delta * d - d) + 4 * (c.max_delta * d + d) + 4 * vecs
    B, T, delta = 1, 816, 9
    io = B * T * dv * 2 + B * delta * A * 4 + 3 * B * c.n_items * d * 4 + B * 4
    assert bench.correction_bytes(c, B, T, delta) == want_w + io


def test_prefill_flops_by_brute_count():
    # Count multiply-adds product by product for a tiny model and compare.
    from synth import GEMMA2B
    cfg = GEMMA2B.with_(n_layers=2, width=8, n_heads=2, head_dim=4, mlp_dim=12)
    B, P = 3, 5
    W, H, D, F = 8, 2, 4, 12
    macs = 0
    for _ in range(cfg.n_layers):
        macs += B * P * W * (H * D + D + D)      # q, k, v
        macs += B * H * P * P * D                # scores
        macs += B * H * P * P * D                # probabilities x V
        macs += B * P * (H * D) * W              # output projection
        macs += B * P * W * F * 2                # gate and up
        macs += B * P * F * W                    # down
    assert bench.prefill_flops(cfg, B, P) == 2 * macs
    # Gemma-2B at 816 tokens: the ~2B projection parameters dominate (3.2 TFLOP per request).
    f = bench.prefill_flops(GEMMA2B, 1, 816)
    assert 3.1e12 < f < 3.4e12
