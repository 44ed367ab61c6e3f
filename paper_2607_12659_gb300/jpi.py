"""ctypes binding of libjpi.so (argument marshalling only).

Every function below calls the C entry point of the same name in ``include/jpi.h``; the
computation runs in the library's CUDA kernels. PyTorch supplies device memory and streams.
If the library has not been built the import of this module still works, but the first call
raises: there is no other implementation to fall back to.
"""

from __future__ import annotations

import ctypes
import os
import re
from ctypes import POINTER, byref, c_float, c_int, c_longlong, c_void_p

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libjpi.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "jpi.h")

JPI_OK = 0
STATUS_NAMES = {
    0: "JPI_OK", -1: "JPI_ERR_INVALID_ARG", -2: "JPI_ERR_SHAPE", -3: "JPI_ERR_OOM",
    -4: "JPI_ERR_CUDA", -5: "JPI_ERR_NOT_READY", -6: "JPI_ERR_DEVICE_TIMEOUT",
    -7: "JPI_ERR_UNSUPPORTED",
}
JPI_BF16, JPI_FP32 = 0, 1

GLOBAL_WEIGHTS = (
    "state_in_w", "state_in_b", "action_in_w", "action_in_b", "action_out_w", "action_out_b",
    "time_mlp_in_w", "time_mlp_in_b", "time_mlp_out_w", "time_mlp_out_b",
    "final_mod_w", "final_mod_b",
)
LAYER_WEIGHTS = (
    "wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down",
    "attn_mod_w", "attn_mod_b", "mlp_mod_w", "mlp_mod_b",
)


class JpiError(RuntimeError):
    def __init__(self, status: int, fn: str, msg: str):
        self.status = status
        super().__init__(f"{fn}: {STATUS_NAMES.get(status, status)}: {msg}")


class jpi_config(ctypes.Structure):
    _fields_ = [(n, c_int) for n in (
        "n_layers", "width", "n_heads", "head_dim", "n_kv_heads", "mlp_dim", "action_dim",
        "state_dim", "time_dim", "max_batch", "max_prefix", "max_chunk", "max_steps")] + [
        ("rope_base", c_float), ("rms_eps", c_float), ("t_min_period", c_float),
        ("t_max_period", c_float), ("precision", c_int)]


class jpi_weights(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in GLOBAL_WEIGHTS + LAYER_WEIGHTS] + [("on_device", c_int)]


_SIGS = {
    "jpi_expert_create": [POINTER(jpi_config), POINTER(jpi_weights), POINTER(c_void_p)],
    "jpi_expert_destroy": [c_void_p],
    "jpi_set_prefix_kv": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p],
    "jpi_prefix_kv_ptr": [c_void_p, c_int, POINTER(c_void_p), POINTER(c_void_p), POINTER(c_longlong)],
    "jpi_commit_prefix": [c_void_p, c_int, c_int],
    "jpi_set_correction": [c_void_p, c_void_p, c_int, c_int, c_void_p],
    "jpi_denoise": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p],
    "jpi_denoise_host": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p],
    "jpi_expert_forward": [c_void_p, c_void_p, c_void_p, c_float, c_int, c_int, c_void_p,
                           c_void_p, c_void_p],
    "jpi_device_status": [c_void_p],
    "jpi_memory_usage": [c_void_p, POINTER(c_longlong)],
    "jpi_graph_kernel_count": [c_void_p, c_int, c_int, c_int, POINTER(c_int)],
    "jpi_profile_op": [c_void_p, c_int, c_int, c_int, c_int, c_int, c_int, c_void_p],
    "jpi_expert_forward_noalloc": [c_void_p, c_void_p, c_void_p, c_float, c_int, c_int, c_void_p,
                                   c_void_p, c_void_p],
}

_lib = None


LIB_HEADERS = ("jpi.h", "jpi_corr.h")   # the entry points libjpi.so exports


def header_symbols(headers=LIB_HEADERS) -> list[str]:
    """Names of every entry point declared in the given headers under include/."""
    inc = os.path.dirname(HEADER)
    names = []
    for f in headers:
        if f.endswith(".h"):
            text = open(os.path.join(inc, f)).read()
            names += re.findall(r"JPI_API\s+[\w\s\*]+?\b(jpi_\w+)\s*\(", text)
    return names


def load():
    """Load libjpi.so (built in-tree by ``build.py``); raise if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is not built: run `python -m paper_2607_12659_gb300.build` "
                           "(the CUDA library is the only implementation)")
    lib = ctypes.CDLL(LIB_PATH)
    for name, args in _SIGS.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = c_int
    lib.jpi_last_error.argtypes = []
    lib.jpi_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(status: int, fn: str):
    if status != JPI_OK:
        raise JpiError(status, fn, load().jpi_last_error().decode(errors="replace"))


def _ptr(t) -> int | None:
    """Raw pointer of a torch tensor or numpy array (None -> NULL)."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


# ------------------------------------------------------------------ thin C-ABI mirrors

def jpi_expert_create(cfg: jpi_config, w: jpi_weights) -> int:
    h = c_void_p()
    _check(load().jpi_expert_create(byref(cfg), byref(w), byref(h)), "jpi_expert_create")
    return h.value


def jpi_expert_destroy(h: int):
    _check(load().jpi_expert_destroy(h), "jpi_expert_destroy")


def jpi_set_prefix_kv(h, k_layers, v_layers, batch, prefix_len, kv_is_fp32, stream=None):
    L = len(k_layers)
    ka = (c_void_p * L)(*[_ptr(k) for k in k_layers])
    va = (c_void_p * L)(*[_ptr(v) for v in v_layers])
    _check(load().jpi_set_prefix_kv(h, ka, va, batch, prefix_len, int(kv_is_fp32), _stream(stream)),
           "jpi_set_prefix_kv")


def jpi_prefix_kv_ptr(h, layer):
    k, v, s = c_void_p(), c_void_p(), c_longlong()
    _check(load().jpi_prefix_kv_ptr(h, layer, byref(k), byref(v), byref(s)), "jpi_prefix_kv_ptr")
    return k.value, v.value, s.value


def jpi_commit_prefix(h, batch, prefix_len):
    _check(load().jpi_commit_prefix(h, batch, prefix_len), "jpi_commit_prefix")


def jpi_set_correction(h, items, batch, num_items, stream=None):
    _check(load().jpi_set_correction(h, _ptr(items), batch, num_items, _stream(stream)),
           "jpi_set_correction")


def jpi_denoise(h, state, noise, batch, chunk, num_steps, out_actions, stream=None):
    _check(load().jpi_denoise(h, _ptr(state), _ptr(noise), batch, chunk, num_steps,
                              _ptr(out_actions), _stream(stream)), "jpi_denoise")


def jpi_denoise_host(h, state, noise, batch, chunk, num_steps, out_actions, stream=None):
    _check(load().jpi_denoise_host(h, _ptr(state), _ptr(noise), batch, chunk, num_steps,
                                   _ptr(out_actions), _stream(stream)), "jpi_denoise_host")


def jpi_expert_forward(h, state, x_t, t, batch, chunk, out_v, out_h=None, stream=None):
    _check(load().jpi_expert_forward(h, _ptr(state), _ptr(x_t), float(t), batch, chunk,
                                     _ptr(out_v), _ptr(out_h), _stream(stream)),
           "jpi_expert_forward")


def jpi_expert_forward_noalloc(h, state, x_t, t, batch, chunk, out_v, out_h=None, stream=None):
    """jpi_expert_forward with its time-conditioning scratch in the library's fixed array."""
    _check(load().jpi_expert_forward_noalloc(h, _ptr(state), _ptr(x_t), float(t), batch, chunk,
                                             _ptr(out_v), _ptr(out_h), _stream(stream)),
           "jpi_expert_forward_noalloc")


def jpi_device_status(h):
    _check(load().jpi_device_status(h), "jpi_device_status")


def jpi_memory_usage(h) -> int:
    b = c_longlong()
    _check(load().jpi_memory_usage(h, byref(b)), "jpi_memory_usage")
    return b.value


def jpi_graph_kernel_count(h, batch, chunk, num_steps) -> int:
    n = c_int()
    _check(load().jpi_graph_kernel_count(h, batch, chunk, num_steps, byref(n)),
           "jpi_graph_kernel_count")
    return n.value


def jpi_profile_op(h, op, layer, batch, chunk, num_steps, reps, stream=None):
    _check(load().jpi_profile_op(h, op, layer, batch, chunk, num_steps, reps, _stream(stream)),
           "jpi_profile_op")


def jpi_last_error() -> str:
    return load().jpi_last_error().decode(errors="replace")


# ------------------------------------------------------------------ convenience wrapper

def make_config(dims, max_batch, max_prefix, max_chunk, max_steps) -> jpi_config:
    """jpi_config from any object with the expert's dimension attributes."""
    return jpi_config(
        n_layers=dims.n_layers, width=dims.width, n_heads=dims.n_heads, head_dim=dims.head_dim,
        n_kv_heads=1, mlp_dim=dims.mlp_dim, action_dim=dims.action_dim,
        state_dim=dims.state_dim, time_dim=dims.time_dim, max_batch=max_batch,
        max_prefix=max_prefix, max_chunk=max_chunk, max_steps=max_steps,
        rope_base=dims.rope_base, rms_eps=dims.rms_eps, t_min_period=dims.t_min_period,
        t_max_period=dims.t_max_period,
        precision=JPI_BF16 if dims.precision == "bf16" else JPI_FP32)


class Expert:
    """A created expert handle; weights are a dict of fp32 host arrays (per-layer lists)."""

    def __init__(self, dims, weights: dict, max_batch=1, max_prefix=1024, max_chunk=64,
                 max_steps=16):
        self.dims = dims
        self.cfg = make_config(dims, max_batch, max_prefix, max_chunk, max_steps)
        keep = []
        wt = jpi_weights(on_device=0)
        for name in GLOBAL_WEIGHTS:
            a = np.ascontiguousarray(weights[name], dtype=np.float32)
            keep.append(a)
            setattr(wt, name, a.ctypes.data)
        for name in LAYER_WEIGHTS:
            arrs = [np.ascontiguousarray(a, dtype=np.float32) for a in weights[name]]
            keep.extend(arrs)
            tab = (c_void_p * len(arrs))(*[a.ctypes.data for a in arrs])
            keep.append(tab)
            setattr(wt, name, ctypes.cast(tab, c_void_p))
        self.handle = jpi_expert_create(self.cfg, wt)
        del keep

    def close(self):
        if self.handle:
            jpi_expert_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_prefix_kv(self, k, v, stream=None):
        """k, v: CUDA tensors [L][B][P][D] (float32 or bfloat16)."""
        import torch
        assert k.is_cuda and v.is_cuda and k.shape == v.shape
        L, B, P, _ = k.shape
        k = k.contiguous()
        v = v.contiguous()
        fp32 = k.dtype == torch.float32
        if not fp32:
            assert k.dtype == torch.bfloat16
        jpi_set_prefix_kv(self.handle, [k[l] for l in range(L)], [v[l] for l in range(L)], B, P,
                          fp32, stream)
        self._kv_keepalive = (k, v)

    def set_correction(self, items, stream=None):
        """items: CUDA float32 tensor [B][T'][width] (T' = 0 clears them), or None to clear."""
        if items is None or items.shape[1] == 0:
            jpi_set_correction(self.handle, None, 1, 0, stream)
            self._corr = None
            self.n_corr = 0
            return
        assert items.is_cuda and items.dim() == 3 and items.shape[2] == self.dims.width
        items = items.contiguous().float()
        B, T, _ = items.shape
        jpi_set_correction(self.handle, items, B, T, stream)
        self._corr = (items,)
        self.n_corr = T

    def denoise(self, state, noise, num_steps, out=None, stream=None):
        import torch
        B, C, _ = noise.shape
        if out is None:
            out = torch.empty_like(noise)
        jpi_denoise(self.handle, state, noise, B, C, num_steps, out, stream)
        return out

    def denoise_host(self, state: np.ndarray, noise: np.ndarray, num_steps: int, out=None,
                     stream=None) -> np.ndarray:
        B, C, _ = noise.shape
        if out is None:
            out = np.empty_like(noise)
        jpi_denoise_host(self.handle, state, noise, B, C, num_steps, out, stream)
        return out

    def forward(self, state, x_t, t, stream=None):
        import torch
        B, C, A = x_t.shape
        v = torch.empty_like(x_t)
        hres = torch.empty((B, 1 + getattr(self, "n_corr", 0) + C, self.dims.width), dtype=torch.float32,
                           device=x_t.device)
        jpi_expert_forward(self.handle, state, x_t, t, B, C, v, hres, stream)
        return v, hres

    def device_status(self):
        jpi_device_status(self.handle)

    def memory_usage(self) -> int:
        return jpi_memory_usage(self.handle)
