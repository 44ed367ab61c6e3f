"""Helpers of the GPU tests: build the library, run the CUDA path, compare with the oracle."""

import json
import os

import pytest

import numpy as np

import oracle
from synth import ExpertConfig

# Tolerances: bf16 weights and tensor-core inputs with fp32 accumulation, and the fp32
# verification mode, against the fp64 oracle on the same (bf16-rounded) inputs.
BF16_MAX_ABS, BF16_REL_L2 = 2e-2, 1e-2
FP32_MAX_ABS = 1e-4

# Small bf16 expert that still spans several 128-row weight tiles and a ragged token tail.
SMALL_BF16 = ExpertConfig(n_layers=2, width=256, n_heads=2, head_dim=128, mlp_dim=512,
                          action_dim=7, state_dim=7, time_dim=64, precision="bf16")

_built = False


def lib():
    global _built
    from paper_2607_12659_gb300 import build, jpi
    if not _built:
        build.build()
        _built = True
    jpi.load()
    return jpi


def to_dev_kv(r, cfg):
    import torch
    dt = torch.bfloat16 if cfg.precision == "bf16" else torch.float32
    return (torch.from_numpy(r["prefix_k"]).cuda().to(dt),
            torch.from_numpy(r["prefix_v"]).cuda().to(dt))


def make_expert(cfg, w, max_batch=1, max_prefix=64, max_chunk=8, max_steps=10):
    return lib().Expert(cfg, w, max_batch=max_batch, max_prefix=max_prefix,
                        max_chunk=max_chunk, max_steps=max_steps)


def gpu_denoise(ex, cfg, r, N):
    import torch
    k, v = to_dev_kv(r, cfg)
    ex.set_prefix_kv(k, v)
    out = ex.denoise(torch.from_numpy(r["state"]).cuda(), torch.from_numpy(r["noise"]).cuda(), N)
    torch.cuda.synchronize()
    ex.device_status()
    return out.cpu().numpy()


def oracle_denoise(cfg, w, r, N, requests=None):
    if requests is None:
        requests = range(r["noise"].shape[0])
    requests = list(requests)
    return oracle.denoise_batch(r["noise"][requests], r["state"][requests], N,
                                r["prefix_k"][:, requests], r["prefix_v"][:, requests], w, cfg)


def errors(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    max_abs = float(np.abs(got - ref).max())
    rel_l2 = float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))
    return max_abs, rel_l2


def log_errors(what, max_abs, rel):
    """Appends one parity record to $JPI_PARITY_LOG (JSON lines) when that is set."""
    path = os.environ.get("JPI_PARITY_LOG")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps({"case": what, "max_abs": max_abs, "rel_l2": rel}) + "\n")


def assert_close(got, ref, cfg, what="", max_abs_tol=None):
    max_abs, rel = errors(got, ref)
    log_errors(what, max_abs, rel)
    if cfg.precision == "bf16":
        tol = BF16_MAX_ABS if max_abs_tol is None else max_abs_tol
        assert max_abs <= tol and rel <= BF16_REL_L2, \
            f"{what}: max-abs {max_abs:.3g} (<= {tol}), rel-L2 {rel:.3g} (<= {BF16_REL_L2})"
    else:
        tol = FP32_MAX_ABS if max_abs_tol is None else max_abs_tol
        assert max_abs <= tol, f"{what}: max-abs {max_abs:.3g} (<= {tol})"
    return max_abs, rel
