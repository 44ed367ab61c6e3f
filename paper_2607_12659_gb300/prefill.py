"""ctypes binding of the LLM prefill's C-ABI (``include/jpi_prefill.h``, ``libjpi_prefill.so``;
argument marshalling only).

``Prefill`` runs the Gemma-shaped prefix prefill on the GPU; ``Prefill.into_expert`` writes every
layer's rotated keys and values straight into an ``Expert``'s KV store (jpi_prefix_kv_ptr) and
commits it (jpi_commit_prefix), so the expert's next denoise attends over them with no copy.
"""

from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, byref, c_float, c_int, c_longlong, c_void_p

import numpy as np

from . import build as _build
from . import jpi
from .jpi import STATUS_NAMES, JpiError, _ptr, _stream

LIB_PATH = _build.PREFILL_LIB
LAYER_WEIGHTS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")


class jpi_prefill_config(ctypes.Structure):
    _fields_ = [(n, c_int) for n in ("n_layers", "width", "n_heads", "head_dim", "mlp_dim", "max_batch",
                                     "max_prefix")] + [("rope_base", c_float), ("rms_eps", c_float)]


class jpi_prefill_weights(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in LAYER_WEIGHTS + ("final_norm",)] + [("on_device", c_int)]


_SIGS = {
    "jpi_prefill_create": [POINTER(jpi_prefill_config), POINTER(jpi_prefill_weights), POINTER(c_void_p)],
    "jpi_prefill_destroy": [c_void_p],
    "jpi_prefill_run": [c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p, c_longlong, c_void_p,
                        c_void_p],
    "jpi_prefill_memory_usage": [c_void_p, POINTER(c_longlong)],
    "jpi_prefill_device_status": [c_void_p],
}

_lib = None


def load():
    """Load libjpi_prefill.so (built in-tree by ``build.py``); raise if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        why = _build.PREFILL_BUILD_ERROR or "run `python -m paper_2607_12659_gb300.build`"
        raise RuntimeError(f"{LIB_PATH} is not built ({why}); the CUDA library is the only implementation")
    lib = ctypes.CDLL(LIB_PATH)
    for name, args in _SIGS.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = c_int
    lib.jpi_prefill_last_error.argtypes = []
    lib.jpi_prefill_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(status: int, fn: str):
    if status != jpi.JPI_OK:
        raise JpiError(status, fn, load().jpi_prefill_last_error().decode(errors="replace"))


def header_symbols() -> list[str]:
    return jpi.header_symbols(("jpi_prefill.h",))


# ------------------------------------------------------------------ thin C-ABI mirrors

def jpi_prefill_create(cfg: jpi_prefill_config, w: jpi_prefill_weights) -> int:
    h = c_void_p()
    _check(load().jpi_prefill_create(byref(cfg), byref(w), byref(h)), "jpi_prefill_create")
    return h.value


def jpi_prefill_destroy(h: int):
    _check(load().jpi_prefill_destroy(h), "jpi_prefill_destroy")


def jpi_prefill_run(h, x, x_is_fp32, batch, prefix_len, k_ptrs, v_ptrs, request_stride, out_final=None,
                    stream=None):
    L = len(k_ptrs)
    ka = (c_void_p * L)(*k_ptrs)
    va = (c_void_p * L)(*v_ptrs)
    _check(load().jpi_prefill_run(h, _ptr(x), int(x_is_fp32), batch, prefix_len, ka, va, request_stride,
                                  _ptr(out_final), _stream(stream)), "jpi_prefill_run")


def jpi_prefill_device_status(h):
    _check(load().jpi_prefill_device_status(h), "jpi_prefill_device_status")


def jpi_prefill_memory_usage(h) -> int:
    b = c_longlong()
    _check(load().jpi_prefill_memory_usage(h, byref(b)), "jpi_prefill_memory_usage")
    return b.value


# ------------------------------------------------------------------ convenience wrapper

def make_prefill_config(dims, max_batch: int, max_prefix: int) -> jpi_prefill_config:
    return jpi_prefill_config(n_layers=dims.n_layers, width=dims.width, n_heads=dims.n_heads,
                              head_dim=dims.head_dim, mlp_dim=dims.mlp_dim, max_batch=max_batch,
                              max_prefix=max_prefix, rope_base=dims.rope_base, rms_eps=dims.rms_eps)


class Prefill:
    """A created prefill handle; weights are a dict of fp32 host arrays (per-layer lists and
    ``final_norm``), named as in ``synth.llm_weight_shapes``."""

    def __init__(self, dims, weights: dict, max_batch: int = 1, max_prefix: int = 1024):
        self.dims = dims
        self.cfg = make_prefill_config(dims, max_batch, max_prefix)
        keep = []
        w = jpi_prefill_weights(on_device=0)
        for name in LAYER_WEIGHTS:
            arrs = [np.ascontiguousarray(a, dtype=np.float32) for a in weights[name]]
            keep.extend(arrs)
            tab = (c_void_p * len(arrs))(*[a.ctypes.data for a in arrs])
            keep.append(tab)
            setattr(w, name, ctypes.cast(tab, c_void_p))
        fn = np.ascontiguousarray(weights["final_norm"], dtype=np.float32)
        keep.append(fn)
        w.final_norm = fn.ctypes.data
        self.handle = jpi_prefill_create(self.cfg, w)
        del keep

    def close(self):
        if self.handle:
            jpi_prefill_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def run(self, x, k_ptrs, v_ptrs, request_stride, final=True, stream=None):
        """x: CUDA tensor [B][P][W] (float32 or bfloat16); k_ptrs / v_ptrs: per-layer device
        addresses of bf16 [B][.][D] destinations (row p of request b at + b request_stride + p D).
        Returns the final-layer output [B][P][W] float32 (or None)."""
        import torch
        assert x.is_cuda and x.dim() == 3 and x.shape[2] == self.dims.width
        x = x.contiguous()
        fp32 = x.dtype == torch.float32
        if not fp32:
            assert x.dtype == torch.bfloat16
        B, P, W = x.shape
        out = torch.empty((B, P, W), dtype=torch.float32, device=x.device) if final else None
        jpi_prefill_run(self.handle, x, fp32, B, P, list(k_ptrs), list(v_ptrs), request_stride, out, stream)
        return out

    def into_tensors(self, x, final=True, stream=None):
        """Runs into fresh bf16 tensors K, V [L][B][P][D]; returns (K, V, final output)."""
        import torch
        B, P, _ = x.shape
        L, D = self.dims.n_layers, self.dims.head_dim
        K = torch.empty((L, B, P, D), dtype=torch.bfloat16, device=x.device)
        V = torch.empty_like(K)
        out = self.run(x, [K[l].data_ptr() for l in range(L)], [V[l].data_ptr() for l in range(L)], P * D,
                       final, stream)
        return K, V, out

    def into_expert(self, x, expert, final=True, stream=None):
        """Writes the KV of every layer into a bf16 Expert's store and commits it."""
        if getattr(expert.dims, "precision", "bf16") != "bf16":
            raise ValueError("the prefill writes bf16 keys and values: the expert must use JPI_BF16")
        B, P, _ = x.shape
        if B > expert.cfg.max_batch or P > expert.cfg.max_prefix:
            raise ValueError(f"batch {B} / prefix {P} exceed the expert store's maxima "
                             f"{expert.cfg.max_batch} / {expert.cfg.max_prefix}")
        if expert.cfg.n_layers != self.dims.n_layers or expert.cfg.head_dim != self.dims.head_dim:
            raise ValueError("the expert's layers and head_dim must match the LLM's")
        ptrs = [jpi.jpi_prefix_kv_ptr(expert.handle, l) for l in range(self.dims.n_layers)]
        stride = ptrs[0][2]
        out = self.run(x, [p[0] for p in ptrs], [p[1] for p in ptrs], stride, final, stream)
        jpi.jpi_commit_prefix(expert.handle, B, P)
        return out

    def device_status(self):
        jpi_prefill_device_status(self.handle)

    def memory_usage(self) -> int:
        return jpi_prefill_memory_usage(self.handle)


__all__ = ["Prefill", "jpi_prefill_create", "jpi_prefill_destroy", "jpi_prefill_run", "jpi_prefill_memory_usage",
           "jpi_prefill_device_status",
           "load", "header_symbols", "STATUS_NAMES"]
