#!/usr/bin/env python
"""Throughput of the flow-matching denoise of the pi0.5-shaped action expert on GB300.

One step = one jpi_denoise call: a full 10-step Euler denoise of one 50 x 32 action chunk at
batch 1 over an 816-token prefix KV (18 layers, width 1024, 8 x 256 heads, GeGLU 4096, bf16
weights). Inputs are seeded synthetic tensors already resident in HBM when the timed region
starts; every call streams 6.2 GB of weights, far more than the 129 MB L2, so no flush is
needed between iterations.

Prints one JSON line (rank 0). `--impl reference` times the fp64 CPU oracle instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "action chunks/s (10-step denoise, batch 1, pi0.5-shaped expert)"
UNIT = "chunks/s"
WORKLOAD = dict(batch=1, prefix=816, chunk=50, steps=10)
WORKLOAD_NAME = ("pi0.5-shaped action expert (18 x W1024, 8x256 heads, 1 KV head, GeGLU 4096), "
                 "batch 1, prefix 816, chunk 50 x 32, 10 Euler steps")
OP_NAMES = {2: "norm+qkv+rope", 3: "attention", 4: "o_proj+residual", 5: "norm+gate_up+geglu",
            6: "down_proj+residual"}

# DRAM bytes per launch from an ncu capture (dram__bytes_read.sum + dram__bytes_write.sum),
# valid only while TRAFFIC_SOURCES hash to `source_sha256`.
NCU_TRAFFIC = {
    # profiles/layer_kernels_pi05_forward.md (layer 1 of one eager forward, batch 1, P 816).
    "norm+qkv+rope": {"bytes": 5489664, "source_sha256": "39321630f8ff0a0e"},
    "attention": {"bytes": 1179648, "source_sha256": "39321630f8ff0a0e"},
    "o_proj+residual": {"bytes": 4695808, "source_sha256": "39321630f8ff0a0e"},
    "norm+gate_up+geglu": {"bytes": 16959744, "source_sha256": "39321630f8ff0a0e"},
    "down_proj+residual": {"bytes": 9131776, "source_sha256": "39321630f8ff0a0e"},
}


# The sources the expert's kernels and their launches are built from. The correction module
# (CORRECTION_SOURCES) is compiled into the same library but none of the measured kernels uses it.
EXPERT_SOURCES = ("api.cu", "attn_t5.cu", "attn_t5_kernel.cuh", "attn_tc.cu", "gemm_big.cuh", "gemm_kernel.cuh",
                  "jpi_internal.h", "kernels_simt.cu", "mod_tc.cu", "noalloc.cu", "ptx.h", "tc_path.cu",
                  "tc_path.h")
CORRECTION_SOURCES = ("corr.cu",)


# The sources the five batch-1 layer kernels of NCU_TRAFFIC are built and launched from (the
# projection kernel, the split-KV attention, their launcher and shared headers): their counters
# stay valid while these are unchanged, whatever changes elsewhere (the large-batch attention).
TRAFFIC_SOURCES = ("attn_tc.cu", "gemm_big.cuh", "gemm_kernel.cuh", "jpi_internal.h", "ptx.h", "tc_path.cu",
                   "tc_path.h")


def source_sha(files=EXPERT_SOURCES) -> str:
    d = os.path.join(ROOT, "paper_2607_12659_gb300", "csrc")
    h = hashlib.sha256()
    for f in sorted(files):
        h.update(open(os.path.join(d, f), "rb").read())
    return h.hexdigest()[:16]


def algorithmic_bytes(cfg, B, P, C, N, items=0):
    """Bytes an ideal denoise must move: weights once per step (bf16), the time/modulation
    weights once per call, the prefix KV once, inputs (with `items` fp32 correction items per
    request) and outputs."""
    W, H, D, F, L, A = cfg.width, cfg.n_heads, cfg.head_dim, cfg.mlp_dim, cfg.n_layers, cfg.action_dim
    per_step = (L * (H * D * W * 2 + 2 * D * W + 3 * F * W) + (cfg.state_dim + 2 * A) * W) * 2
    time_w = (W * cfg.time_dim + W * W + (6 * L + 2) * W * W) * 2
    kv = B * L * P * D * 2 * 2
    io = B * (cfg.state_dim + 2 * C * A + items * W) * 4
    return N * per_step + time_w + kv + io


def algorithmic_flops(cfg, B, P, C, N, items=0):
    """Multiply-adds x 2 of a denoise: the layer projections at M = B (C + 1 + items) tokens, the
    attention of the S H query rows over all P + S keys (QK^T and PV), the state/action
    embeddings and the action-out projection, and per step time the time MLP and the
    modulation GEMV."""
    W, H, D, F, L = cfg.width, cfg.n_heads, cfg.head_dim, cfg.mlp_dim, cfg.n_layers
    Sd, A = cfg.state_dim, cfg.action_dim
    S = C + 1 + items
    Mt = B * S
    proj = L * (H * D * W + 2 * D * W + H * D * W + 3 * F * W)
    attn = L * B * S * H * (P + S) * D * 2
    per_step = 2 * (Mt * proj + attn + B * Sd * W + B * C * A * W + B * C * W * A)
    per_time = 2 * (W * cfg.time_dim + W * W + (6 * L + 2) * W * W)
    return N * (per_step + per_time)


def op_bytes(cfg, op, B, P, C, items=0):
    """Algorithmic bytes of one launch of a layer op (weights + activation reads/writes)."""
    W, H, D, F = cfg.width, cfg.n_heads, cfg.head_dim, cfg.mlp_dim
    Mt = B * (C + 1 + items)
    if op == 2:
        return (H + 2) * D * W * 2 + Mt * W * 4 + Mt * (H + 2) * D * 2
    if op == 3:
        return B * (P + C + 1 + items) * D * 2 * 2 + Mt * H * D * 2 * 2
    if op == 4:
        return W * H * D * 2 + Mt * H * D * 2 + Mt * W * 4 * 2
    if op == 5:
        return 2 * F * W * 2 + Mt * W * 4 + Mt * F * 2
    if op == 6:
        return F * W * 2 + Mt * F * 2 + Mt * W * 4 * 2
    raise ValueError(op)


def rank_env():
    """(world size, rank, local rank) from the launcher's environment; (1, 0, 0) when run directly."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x: float, world: int, device) -> float:
    """The slowest rank's value (max-over-ranks timing); x itself at world size 1."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, batch: int, steps: int, ms: float) -> float:
    """Chunks per second of the whole job: every replica denoises `steps` batches of `batch`
    requests in `ms` milliseconds (the slowest replica's time)."""
    return world * batch * steps / (ms / 1e3)


def request_seed(rank: int) -> int:
    """Seed of a replica's requests: each rank denoises its own, independent requests."""
    return 2001 + rank


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d.get("bf16_tflops"), "measured"
    return 6800.0, 1900.0, "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle samples every 50 ms while the timed region runs. The region
    starts only after the first sample has arrived, so the samples cover all of it."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def _read(self):
        for line in self.proc.stdout:
            if line.strip():
                self.lines.append(line)
                self.first.set()
        self.first.set()

    def __enter__(self):
        import threading
        self.lines = []
        self.first = threading.Event()
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return self
        self.reader = threading.Thread(target=self._read, daemon=True)
        self.reader.start()
        self.first.wait(timeout=5.0)
        self.n_before = len(self.lines)
        return self

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.proc.wait()
            self.reader.join(timeout=5)
            # Samples taken during the region (the one that opened it included).
            self.lines = self.lines[max(self.n_before - 1, 0):]

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in getattr(self, "lines", []):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def cpu_baseline_child():
    """Times the fp64 oracle on one full request of the workload (runs in a subprocess whose
    BLAS thread count is fixed by the parent)."""
    import numpy as np
    import oracle
    from synth import PI05, make_requests, make_weights
    B, P, C, N = (WORKLOAD[k] for k in ("batch", "prefix", "chunk", "steps"))
    w = oracle.to_f64(make_weights(PI05, 2000))
    r = make_requests(PI05, 2001, 1, P, C)
    args = (r["prefix_k"][:, 0].astype(np.float64), r["prefix_v"][:, 0].astype(np.float64), w, PI05)
    oracle.expert_forward(r["noise"][0].astype(np.float64), r["state"][0].astype(np.float64), 0.0, *args)
    t0 = time.perf_counter()
    oracle.denoise(r["noise"][0], r["state"][0].astype(np.float64), N, *args)
    dt = time.perf_counter() - t0
    print(json.dumps({"seconds": dt}))


def run_cpu_baseline(cores: int) -> dict:
    env = dict(os.environ, OPENBLAS_NUM_THREADS=str(cores), OMP_NUM_THREADS=str(cores),
               MKL_NUM_THREADS=str(cores))
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-baseline-child"],
                       capture_output=True, text=True, env=env, timeout=900)
    if r.returncode != 0:
        return {"value": None, "unit": UNIT, "cores": cores, "kind": "oracle",
                "sample": "failed: " + r.stderr.strip().splitlines()[-1][:200] if r.stderr else "failed"}
    sec = json.loads(r.stdout.strip().splitlines()[-1])["seconds"]
    return {"value": 1.0 / sec, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"one full request: 10-step denoise at batch 1 (P 816, C 50), fp64 numpy "
                      f"oracle, {sec:.2f} s"}


def reference_arm(args):
    """The fp64 CPU oracle on this host's cores; a step is one Euler step (one expert pass)
    of the batch-1 workload, and chunks/s = 1 / (10 x mean step time)."""
    _, rank, _ = rank_env()
    if rank != 0:
        return
    import numpy as np
    import oracle
    from synth import PI05, make_requests, make_weights
    cores = os.cpu_count() or 1
    B, P, C, N = (WORKLOAD[k] for k in ("batch", "prefix", "chunk", "steps"))
    w = oracle.to_f64(make_weights(PI05, 2000))
    r = make_requests(PI05, 2001, 1, P, C)
    a = (r["prefix_k"][:, 0].astype(np.float64), r["prefix_v"][:, 0].astype(np.float64), w, PI05)
    x, s = r["noise"][0].astype(np.float64), r["state"][0].astype(np.float64)
    times = []
    for i in range(args.warmup + args.steps):
        t = (i % N) / N
        t0 = time.perf_counter()
        x = x + (1.0 / N) * oracle.expert_forward(x, s, t, *a)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    step = statistics.mean(times)
    value = 1.0 / (N * step)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_NAME, **WORKLOAD,
                   "reference_step": "one Euler step (one expert pass) of the workload"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{args.steps} Euler steps of one batch-1 request, fp64 numpy oracle"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def our_arm(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2607_12659_gb300 import build, jpi
    from synth import PI05, make_correction, make_requests, make_weights

    world, rank, local = rank_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        build.build()
    if world > 1:
        dist.barrier()
    jpi.load()

    B, P, C, N = (WORKLOAD[k] for k in ("batch", "prefix", "chunk", "steps"))
    B, P = args.batch or B, args.prefix or P
    default_workload = (B, P) == (WORKLOAD["batch"], WORKLOAD["prefix"]) and not args.items
    cfg = PI05
    w = make_weights(cfg, 2000)
    ex = jpi.Expert(cfg, w, max_batch=B, max_prefix=P, max_chunk=C, max_steps=N)
    del w
    r = make_requests(cfg, request_seed(rank), B, P, C)
    ex.set_prefix_kv(torch.from_numpy(r["prefix_k"]).cuda().to(torch.bfloat16),
                     torch.from_numpy(r["prefix_v"]).cuda().to(torch.bfloat16))
    if args.items:
        # The correction items of Sec. 4.1 as context tokens (T' = 4 in App. B).
        ex.set_correction(torch.from_numpy(make_correction(cfg, request_seed(rank) + 1, B, args.items)).cuda())
    state = torch.from_numpy(r["state"]).cuda()
    noise = torch.from_numpy(r["noise"]).cuda()
    out = torch.empty_like(noise)
    stream = torch.cuda.current_stream()

    t0 = time.perf_counter()
    ex.denoise(state, noise, N, out)              # first call captures the graph
    torch.cuda.synchronize()
    capture_s = time.perf_counter() - t0
    for _ in range(max(args.warmup - 1, 0)):
        ex.denoise(state, noise, N, out)
    torch.cuda.synchronize()
    ex.device_status()

    # ---- timed region: K denoise calls, device events on the launching stream ----
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        evs[0].record(stream)
        for i in range(args.steps):
            ex.denoise(state, noise, N, out)
            evs[i + 1].record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    per = [evs[i].elapsed_time(evs[i + 1]) for i in range(args.steps)]
    total_ms = evs[0].elapsed_time(evs[-1])
    ex.device_status()
    t_max = max_over_ranks(total_ms, world, "cuda")
    ms_per_step = t_max / args.steps
    value = whole_job_rate(world, B, args.steps, t_max)

    # ---- end to end through the host-buffer entry point (pinned host memory) ----
    hs = torch.from_numpy(r["state"]).pin_memory()
    hn = torch.from_numpy(r["noise"]).pin_memory()
    ho = torch.empty_like(hn).pin_memory()
    hs_np, hn_np, ho_np = hs.numpy(), hn.numpy(), ho.numpy()
    for _ in range(2):
        ex.denoise_host(hs_np, hn_np, N, ho_np)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        ex.denoise_host(hs_np, hn_np, N, ho_np)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, "cuda")
    e2e_value = whole_job_rate(world, B, args.steps, e2e_ms)
    same = bool(np.array_equal(ho_np, out.cpu().numpy()))

    # ---- per-op durations (each op alone, back to back, events on the launching stream) ----
    reps = 20
    op_ms = {}
    for op in OP_NAMES:
        jpi.jpi_profile_op(ex.handle, op, 0, B, C, N, 3, stream)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        jpi.jpi_profile_op(ex.handle, op, 0, B, C, N, reps, stream)
        b.record(stream)
        torch.cuda.synchronize()
        op_ms[op] = a.elapsed_time(b) / reps
    dom = max(op_ms, key=op_ms.get)
    hbm_peak, tc_peak, peak_src = measured_peaks()
    dom_bytes = op_bytes(cfg, dom, B, P, C, args.items)
    achieved = dom_bytes / (op_ms[dom] * 1e-3) / 1e9
    sha = source_sha()
    tr = NCU_TRAFFIC.get(OP_NAMES[dom])
    traffic = (tr["bytes"] if tr and tr.get("source_sha256") == source_sha(TRAFFIC_SOURCES) and default_workload
               else None)

    n_kernels = jpi.jpi_graph_kernel_count(ex.handle, B, C, N)
    alg = algorithmic_bytes(cfg, B, P, C, N, args.items)
    path_bw = alg / (ms_per_step * 1e-3) / 1e9
    flops = algorithmic_flops(cfg, B, P, C, N, args.items)
    path_tf = flops / (ms_per_step * 1e-3) / 1e12

    if rank == 0:
        cpu = None
        if world == 1 and default_workload and not args.no_cpu_baseline:
            cpu = run_cpu_baseline(os.cpu_count() or 1)
            one = run_cpu_baseline(1)          # the same oracle on one thread
            cpu["single_thread"] = {"value": one["value"], "cores": 1, "sample": one["sample"]}
        clocks = clk.summary()
        line = {
            "metric": METRIC if default_workload else METRIC.replace("batch 1", f"batch {B}"),
            "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD_NAME if default_workload else
                       WORKLOAD_NAME.replace("batch 1, prefix 816", f"batch {B}, prefix {P}")
                       + (f", {args.items} correction items" if args.items else ""),
                       **WORKLOAD, "batch": B, "prefix": P, "correction_items": args.items,
                       "l2": "no flush: each call streams 6.2 GB of weights (> 129 MB L2)",
                       "parallelism": f"replicas x{world}"},
            "us_per_denoise": {"median": statistics.median(per) * 1e3,
                               "p10": sorted(per)[max(0, int(0.1 * len(per)) - 0)] * 1e3,
                               "p90": sorted(per)[min(len(per) - 1, int(0.9 * len(per)))] * 1e3},
            "path_roofline": {"bound": "hbm", "algorithmic_bytes": alg, "achieved_gbs": path_bw,
                              "peak_gbs": hbm_peak, "frac": path_bw / hbm_peak,
                              "roofline_us": alg / hbm_peak / 1e3,
                              "algorithmic_flops": flops, "achieved_tflops": path_tf,
                              "tensor_peak_tflops": tc_peak, "tensor_frac": path_tf / tc_peak if tc_peak else None},
            "roofline": {"bound": "hbm", "kernel": OP_NAMES[dom], "achieved": achieved,
                         "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
                         "traffic": traffic, "peak_source": peak_src,
                         "bytes_per_launch": dom_bytes, "us_per_launch": op_ms[dom] * 1e3},
            "op_us": {OP_NAMES[k]: v * 1e3 for k, v in op_ms.items()},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT,
                    "h2d_bytes_per_step": int(hs.numel() * 4 + hn.numel() * 4),
                    "d2h_bytes_per_step": int(ho.numel() * 4), "matches_device_path": same},
            "gpu_launches": n_kernels * args.steps,
            "kernels_per_denoise": n_kernels,
            "graph_capture_s": capture_s,
            "clocks": clocks,
            "source_sha256": sha,
        }
        print(json.dumps(line), flush=True)
    ex.close()
    if world > 1:
        dist.destroy_process_group()


# Correction-module tensors used only at create time (the compressor's query self-attention and
# the cross-attention queries mapped through the key projection): not streamed per call.
CORR_CREATE_ONLY = ("qf_query", "qf_ln1_w", "qf_ln1_b", "qf_ln2_w", "qf_ln2_b", "qf_ca_wq", "qf_ca_bq",
                    "qf_ca_wk", "qf_ca_bk")


def correction_bytes(cfg, B, T, delta):
    """Bytes one compress + predict call must move: every per-call weight once (projection
    matrices in bf16; vectors, the position table and the confidence row in fp32, as the library
    stores them), the bf16 VLM output, the actions, the state in and out, the confidences."""
    import numpy as np
    from synth.correction import correction_weight_shapes
    wb = 0
    for name, shp in correction_weight_shapes(cfg).items():
        if name in CORR_CREATE_ONLY or name.startswith("qf_sa_"):
            continue
        mat = len(shp) == 2 and name not in ("act_pos", "conf_w")
        wb += int(np.prod(shp)) * (2 if mat and cfg.precision == "bf16" else 4)
    io = B * T * cfg.d_vlm * 2 + B * delta * cfg.action_dim * 4 + 3 * B * cfg.n_items * cfg.width * 4 + B * 4
    return wb + io


def correction_arm(args):
    """The future correction module (compress + predict, pi0.5 sizes, bf16 weights) timed alone."""
    import torch
    from paper_2607_12659_gb300 import build, corr
    from synth.correction import PI05_CORRECTION, make_correction_inputs, make_correction_weights
    build.build()
    torch.cuda.set_device(0)
    cfg = PI05_CORRECTION
    B, T, delta = args.batch or 1, args.prefix or WORKLOAD["prefix"], 9
    mod = corr.Corrector(cfg, make_correction_weights(cfg, 3000), max_batch=B, max_vlm_tokens=T)
    inp = make_correction_inputs(cfg, 3001, B, T, delta)
    hv = torch.from_numpy(inp["h_vlm"]).cuda().to(torch.bfloat16)
    acts = torch.from_numpy(inp["actions"]).cuda()
    state = torch.empty((B, cfg.n_items, cfg.width), dtype=torch.float32, device="cuda")
    hf, conf = torch.empty_like(state), torch.empty((B,), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        mod.compress(hv, out=state)
        mod.predict(state, acts, out=hf, confidence=conf)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3 * args.steps)]
    with ClockSampler(0) as clk:
        for i in range(args.steps):
            ev[3 * i].record(stream)
            mod.compress(hv, out=state)
            ev[3 * i + 1].record(stream)
            mod.predict(state, acts, out=hf, confidence=conf)
            ev[3 * i + 2].record(stream)
        torch.cuda.synchronize()
    comp = [ev[3 * i].elapsed_time(ev[3 * i + 1]) for i in range(args.steps)]
    pred = [ev[3 * i + 1].elapsed_time(ev[3 * i + 2]) for i in range(args.steps)]
    call_ms = statistics.median([a + b for a, b in zip(comp, pred)])
    hbm_peak, _, peak_src = measured_peaks()
    alg = correction_bytes(cfg, B, T, delta)
    achieved = alg / (call_ms * 1e-3) / 1e9
    print(json.dumps({
        "metric": f"future correction module calls/s (compress + predict), batch {B}",
        "value": B / (call_ms * 1e-3), "unit": "calls/s", "steps": args.steps, "warmup": args.warmup,
        "config": {"workload": f"pi0.5-sized correction module (d_AE 1024, d_VLM 2048, T' 4), "
                               f"{T} VLM tokens, Delta {delta}", "batch": B},
        "us": {"compress": statistics.median(comp) * 1e3, "predict": statistics.median(pred) * 1e3,
               "call": call_ms * 1e3},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "traffic": None, "peak_source": peak_src,
                     "bytes_per_call": alg},
        "dtype": "bf16 weights, fp32 activations", "data": "synthetic", "clocks": clk.summary(),
    }), flush=True)
    mod.close()


def prefill_flops(cfg, B, P):
    """FLOPs of one prefill: 2 per multiply-add of every projection (Q/K/V, output, gate/up, down)
    over B P tokens, plus the scores and the probability-weighted values (H P^2 D each) per
    request and layer."""
    W, H, D, F = cfg.width, cfg.n_heads, cfg.head_dim, cfg.mlp_dim
    proj = W * (H + 2) * D + H * D * W + 2 * F * W + F * W
    return cfg.n_layers * (2 * B * P * proj + 2 * 2 * B * H * P * P * D)


def prefill_arm(args):
    """The Gemma-2B-shaped prefill (18 layers, bf16 weights) timed alone, into KV tensors."""
    import torch
    from paper_2607_12659_gb300 import build, prefill
    from synth import GEMMA2B, make_llm_weights, make_prefix_embeddings
    build.build()
    torch.cuda.set_device(0)
    cfg = GEMMA2B
    B, P = args.batch or 1, args.prefix or WORKLOAD["prefix"]
    pre = prefill.Prefill(cfg, make_llm_weights(cfg, 4000), max_batch=B, max_prefix=P)
    x = torch.from_numpy(make_prefix_embeddings(cfg, 4001, B, P)).cuda().to(torch.bfloat16)
    L, D = cfg.n_layers, cfg.head_dim
    K = torch.empty((L, B, P, D), dtype=torch.bfloat16, device="cuda")
    V = torch.empty_like(K)
    kp, vp = [K[l].data_ptr() for l in range(L)], [V[l].data_ptr() for l in range(L)]
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        pre.run(x, kp, vp, P * D, final=False)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    with ClockSampler(0) as clk:
        ev[0].record(stream)
        for i in range(args.steps):
            pre.run(x, kp, vp, P * D, final=False)
            ev[i + 1].record(stream)
        torch.cuda.synchronize()
    ms = statistics.median([ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)])
    _, tc_peak, peak_src = measured_peaks()
    flops = prefill_flops(cfg, B, P)
    tf = flops / (ms * 1e-3) / 1e12
    print(json.dumps({
        "metric": f"Gemma-2B prefix prefill, {P} tokens x batch {B}, ms per prefill",
        "value": ms, "unit": "ms", "higher_is_better": False, "steps": args.steps, "warmup": args.warmup,
        "config": {"workload": f"Gemma-2B-shaped LLM (18 x W2048, 8x256 heads, 1 KV head, GeGLU 16384), "
                               f"batch {B}, prefix {P}"},
        "roofline": {"bound": "tensor", "achieved": tf, "peak": tc_peak, "unit": "TFLOP/s",
                     "frac": tf / tc_peak if tc_peak else None, "traffic": None, "peak_source": peak_src,
                     "flops_per_call": flops},
        "dtype": "bf16 GEMM operands, fp32 accumulation and residual stream", "data": "synthetic",
        "clocks": clk.summary(),
    }), flush=True)
    pre.close()


SWEEP = dict(prefix=(256, 512, 816, 1536), chunk=(10, 50), steps=(1, 5, 10))


def sweep_arm(args):
    """The batch-1 sweep over prefix length, chunk length and Euler steps (24 cases) in one
    process: one expert sized for the largest case, a graph per case (captured on its first
    call, untimed), then `--steps` timed calls. One JSON line with every case's median time
    against its HBM roofline (a table beside the bench line, not a bench line)."""
    import torch
    from paper_2607_12659_gb300 import build, jpi
    from synth import PI05, make_requests, make_weights
    build.build()
    jpi.load()
    torch.cuda.set_device(0)
    cfg = PI05
    ex = jpi.Expert(cfg, make_weights(cfg, 2000), max_batch=1, max_prefix=max(SWEEP["prefix"]),
                    max_chunk=max(SWEEP["chunk"]), max_steps=max(SWEEP["steps"]))
    hbm_peak, _, peak_src = measured_peaks()
    stream = torch.cuda.current_stream()
    cases = []
    with ClockSampler(0) as clk:
        for P in SWEEP["prefix"]:
            for C in SWEEP["chunk"]:
                r = make_requests(cfg, 3000 + P + C, 1, P, C)
                ex.set_prefix_kv(torch.from_numpy(r["prefix_k"]).cuda().to(torch.bfloat16),
                                 torch.from_numpy(r["prefix_v"]).cuda().to(torch.bfloat16))
                state = torch.from_numpy(r["state"]).cuda()
                noise = torch.from_numpy(r["noise"]).cuda()
                out = torch.empty_like(noise)
                for N in SWEEP["steps"]:
                    for _ in range(args.warmup):
                        ex.denoise(state, noise, N, out)
                    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
                    torch.cuda.synchronize()
                    ev[0].record(stream)
                    for i in range(args.steps):
                        ex.denoise(state, noise, N, out)
                        ev[i + 1].record(stream)
                    torch.cuda.synchronize()
                    ex.device_status()
                    us = statistics.median([ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)]) * 1e3
                    roof_us = algorithmic_bytes(cfg, 1, P, C, N) / (hbm_peak * 1e9) * 1e6
                    cases.append({"prefix": P, "chunk": C, "steps": N, "us_per_denoise": round(us, 1),
                                  "chunks_per_s": round(1e6 / us, 1), "roofline_us": round(roof_us, 1),
                                  "frac": round(roof_us / us, 4)})
    print(json.dumps({
        "metric": "us per denoise, batch 1, prefix x chunk x Euler-step sweep (pi0.5-shaped expert)",
        "cases": cases, "steps": args.steps, "warmup": args.warmup,
        "roofline": {"bound": "hbm", "peak": hbm_peak, "unit": "GB/s", "peak_source": peak_src},
        "dtype": "bf16 GEMM operands, fp32 accumulation and residual stream", "data": "synthetic",
        "clocks": clk.summary(),
    }), flush=True)
    ex.close()


def profile_forward(args):
    """Small case for kernel captures: the workload's expert, eager expert passes (batch and
    prefix as given, else the workload's)."""
    import torch
    from paper_2607_12659_gb300 import build, jpi
    from synth import PI05, make_requests, make_weights
    build.build()
    jpi.load()
    torch.cuda.set_device(0)
    B, P, C = args.batch or WORKLOAD["batch"], args.prefix or WORKLOAD["prefix"], WORKLOAD["chunk"]
    ex = jpi.Expert(PI05, make_weights(PI05, 2000), max_batch=B, max_prefix=P, max_chunk=C,
                    max_steps=WORKLOAD["steps"])
    r = make_requests(PI05, 2001, B, P, C)
    ex.set_prefix_kv(torch.from_numpy(r["prefix_k"]).cuda().to(torch.bfloat16),
                     torch.from_numpy(r["prefix_v"]).cuda().to(torch.bfloat16))
    s, x = torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda()
    for _ in range(args.forward_passes):
        ex.forward(s, x, 0.0)
    torch.cuda.synchronize()
    ex.device_status()
    print(json.dumps({"profile_forward": "ok", "passes": args.forward_passes}))


def primitives_arm():
    """The hardware-primitive costs that bound the denoise (csrc/probe/primitives.cu): hand-offs
    behind the batch-1 chain, per-SM operand intake behind large batches. One JSON line (a
    diagnostic, not a bench line)."""
    from paper_2607_12659_gb300 import build
    binary = build.build_probe()
    r = subprocess.run([binary], capture_output=True, text=True, timeout=300)
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    if r.returncode != 0 or not lines:
        raise SystemExit(f"primitives probe failed ({r.returncode}): {r.stdout[-400:]} {r.stderr[-400:]}")
    out = json.loads(lines[-1])
    print(json.dumps({"metric": "GB300 primitive costs behind the denoise (diagnostic)",
                      "primitives": out, "clocks_note": "not sampled; durations are medians of short loops"}),
          flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--primitives", action="store_true",
                    help="measure the hand-off, barrier, reduction, copy and MMA-issue costs (diagnostic)")
    ap.add_argument("--profile-forward", action="store_true",
                    help="run eager expert passes of the workload (small case for ncu captures)")
    ap.add_argument("--forward-passes", type=int, default=2)
    ap.add_argument("--correction", action="store_true",
                    help="time the future correction module alone (compress + predict)")
    ap.add_argument("--prefill", action="store_true", help="time the Gemma-2B-shaped prefix prefill alone")
    ap.add_argument("--sweep", action="store_true",
                    help="time the batch-1 prefix x chunk x Euler-step sweep (24 cases, one JSON line)")
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="requests per denoise (default: the batch-1 workload); for documentation runs")
    ap.add_argument("--prefix", type=int, default=0, help="prefix tokens per request (default 816)")
    ap.add_argument("--items", type=int, default=0,
                    help="correction items (context tokens) per request, 0..8; for documentation runs")
    ap.add_argument("--cpu-baseline-child", action="store_true", help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.cpu_baseline_child:
        cpu_baseline_child()
        return
    if args.profile_forward:
        profile_forward(args)
        return
    if args.primitives:
        primitives_arm()
        return
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.correction:
        correction_arm(args)
    elif args.prefill:
        prefill_arm(args)
    elif args.sweep:
        sweep_arm(args)
    elif args.impl == "reference":
        reference_arm(args)
    else:
        our_arm(args)


if __name__ == "__main__":
    main()
