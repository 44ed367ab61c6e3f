"""ctypes binding of the future correction module's C-ABI (``include/jpi_corr.h``; argument
marshalling only).

Every ``jpi_corr_*`` function below calls the library entry point of the same name; the
computation runs in the library's CUDA kernels (``csrc/corr.cu``). ``Corrector`` wraps a handle
for PyTorch CUDA tensors: ``compress`` turns the VLM's final-layer output into the compressed
state (App. B's Q-Former), ``predict`` runs f_corr of Alg. 1 on a compressed state and the
committed actions and returns the predicted state (the expert's correction items, see
``Expert.set_correction``) with its confidence.
"""

from __future__ import annotations

import ctypes
from ctypes import POINTER, byref, c_float, c_int, c_longlong, c_void_p

import numpy as np

from . import jpi
from .jpi import JPI_BF16, JPI_FP32, _check, _ptr, _stream

BLOCK_FIELDS = ("ln1_w", "ln1_b", "wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo",
                "ln2_w", "ln2_b", "w1", "b1", "w2", "b2")


class jpi_corr_config(ctypes.Structure):
    _fields_ = [(n, c_int) for n in (
        "width", "n_heads", "head_dim", "mlp_dim", "d_vlm", "n_items", "action_dim", "max_delta",
        "n_joint", "max_batch", "max_vlm_tokens")] + [("ln_eps", c_float), ("precision", c_int)]


class jpi_corr_block(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in BLOCK_FIELDS]


def _p(*names):
    return [(n, c_void_p) for n in names]


class jpi_corr_weights(ctypes.Structure):
    _fields_ = (_p("qf_query") + [("qf_sa", jpi_corr_block)] + _p("qf_ln2_w", "qf_ln2_b")
                + _p("qf_ca_wq", "qf_ca_bq", "qf_ca_wk", "qf_ca_bk", "qf_ca_wv", "qf_ca_bv",
                     "qf_ca_wo", "qf_ca_bo")
                + _p("qf_ln3_w", "qf_ln3_b", "qf_mlp_w1", "qf_mlp_b1", "qf_mlp_w2", "qf_mlp_b2")
                + _p("qf_lnf_w", "qf_lnf_b")
                + _p("act_w1", "act_b1", "act_w2", "act_b2", "act_pos") + [("ab", jpi_corr_block)]
                + _p("fuse_w", "fuse_b") + [("jb", POINTER(jpi_corr_block))]
                + _p("head_ln_w", "head_ln_b", "corr_w", "corr_b", "conf_w", "conf_b")
                + [("on_device", c_int)])


_SIGS = {
    "jpi_corr_create": [POINTER(jpi_corr_config), POINTER(jpi_corr_weights), POINTER(c_void_p)],
    "jpi_corr_destroy": [c_void_p],
    "jpi_corr_compress": [c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p],
    "jpi_corr_predict": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_void_p, c_void_p, c_void_p],
    "jpi_corr_memory_usage": [c_void_p, POINTER(c_longlong)],
}


def load():
    """The library (built in-tree), with the correction module's signatures set."""
    lib = jpi.load()
    for name, args in _SIGS.items():
        fn = getattr(lib, name)
        if fn.argtypes != args:
            fn.argtypes = args
            fn.restype = c_int
    return lib


# ------------------------------------------------------------------ thin C-ABI mirrors

def jpi_corr_create(cfg: jpi_corr_config, w: jpi_corr_weights) -> int:
    h = c_void_p()
    _check(load().jpi_corr_create(byref(cfg), byref(w), byref(h)), "jpi_corr_create")
    return h.value


def jpi_corr_destroy(h: int):
    _check(load().jpi_corr_destroy(h), "jpi_corr_destroy")


def jpi_corr_compress(h, h_vlm, vlm_is_fp32, batch, n_tokens, out_state, stream=None):
    _check(load().jpi_corr_compress(h, _ptr(h_vlm), int(vlm_is_fp32), batch, n_tokens, _ptr(out_state),
                                    _stream(stream)), "jpi_corr_compress")


def jpi_corr_predict(h, state, actions, batch, delta, out_state, out_confidence=None, stream=None):
    _check(load().jpi_corr_predict(h, _ptr(state), _ptr(actions), batch, delta, _ptr(out_state),
                                   _ptr(out_confidence), _stream(stream)), "jpi_corr_predict")


def jpi_corr_memory_usage(h) -> int:
    b = c_longlong()
    _check(load().jpi_corr_memory_usage(h, byref(b)), "jpi_corr_memory_usage")
    return b.value


# ------------------------------------------------------------------ convenience wrapper

def make_corr_config(dims, max_batch: int, max_vlm_tokens: int) -> jpi_corr_config:
    """jpi_corr_config from any object with the module's dimension attributes."""
    return jpi_corr_config(
        width=dims.width, n_heads=dims.n_heads, head_dim=dims.head_dim, mlp_dim=dims.mlp_dim,
        d_vlm=dims.d_vlm, n_items=dims.n_items, action_dim=dims.action_dim,
        max_delta=dims.max_delta, n_joint=dims.n_joint, max_batch=max_batch,
        max_vlm_tokens=max_vlm_tokens, ln_eps=dims.ln_eps,
        precision=JPI_BF16 if dims.precision == "bf16" else JPI_FP32)


class Corrector:
    """A created correction-module handle; weights are a dict of fp32 host arrays named as in
    ``synth.correction_weight_shapes`` (qf_*, act_*, ab_*, fuse_*, jb{i}_*, head_ln, corr_*,
    conf_*)."""

    def __init__(self, dims, weights: dict, max_batch: int = 1, max_vlm_tokens: int = 1024):
        self.dims = dims
        self.cfg = make_corr_config(dims, max_batch, max_vlm_tokens)
        keep = []

        def ptr(name):
            a = np.ascontiguousarray(weights[name], dtype=np.float32).reshape(-1)
            keep.append(a)
            return a.ctypes.data

        def block(prefix, attn_prefix, with_mlp=True):
            b = jpi_corr_block()
            b.ln1_w, b.ln1_b = ptr(prefix + "ln1_w"), ptr(prefix + "ln1_b")
            for f in ("wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo"):
                setattr(b, f, ptr(attn_prefix + f))
            if with_mlp:
                b.ln2_w, b.ln2_b = ptr(prefix + "ln2_w"), ptr(prefix + "ln2_b")
                for f in ("w1", "b1", "w2", "b2"):
                    setattr(b, f, ptr(prefix + "mlp_" + f))
            return b

        w = jpi_corr_weights(on_device=0)
        w.qf_query = ptr("qf_query")
        w.qf_sa = block("qf_", "qf_sa_", with_mlp=False)
        for name in ("qf_ln2_w", "qf_ln2_b", "qf_ca_wq", "qf_ca_bq", "qf_ca_wk", "qf_ca_bk",
                     "qf_ca_wv", "qf_ca_bv", "qf_ca_wo", "qf_ca_bo", "qf_ln3_w", "qf_ln3_b",
                     "qf_mlp_w1", "qf_mlp_b1", "qf_mlp_w2", "qf_mlp_b2", "qf_lnf_w", "qf_lnf_b",
                     "act_w1", "act_b1", "act_w2", "act_b2", "act_pos", "fuse_w", "fuse_b",
                     "head_ln_w", "head_ln_b", "corr_w", "corr_b", "conf_w", "conf_b"):
            setattr(w, name, ptr(name))
        w.ab = block("ab_", "ab_sa_")
        n = dims.n_joint
        jb = (jpi_corr_block * max(n, 1))(*[block(f"jb{i}_", f"jb{i}_sa_") for i in range(n)])
        keep.append(jb)
        w.jb = ctypes.cast(jb, POINTER(jpi_corr_block)) if n else None
        self.handle = jpi_corr_create(self.cfg, w)
        del keep

    def close(self):
        if self.handle:
            jpi_corr_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def compress(self, h_vlm, out=None, stream=None):
        """h_vlm: CUDA tensor [B][T][d_vlm], float32 or bfloat16 -> [B][T'][width] float32."""
        import torch
        assert h_vlm.is_cuda and h_vlm.dim() == 3 and h_vlm.shape[2] == self.dims.d_vlm
        h_vlm = h_vlm.contiguous()
        fp32 = h_vlm.dtype == torch.float32
        if not fp32:
            assert h_vlm.dtype == torch.bfloat16
        B, T, _ = h_vlm.shape
        if out is None:
            out = torch.empty((B, self.dims.n_items, self.dims.width), dtype=torch.float32,
                              device=h_vlm.device)
        jpi_corr_compress(self.handle, h_vlm, fp32, B, T, out, stream)
        return out

    def predict(self, state, actions, out=None, confidence=None, stream=None):
        """state [B][T'][width], actions [B][delta][A] (CUDA float32) -> (predicted state
        [B][T'][width], confidence [B])."""
        import torch
        assert state.is_cuda and actions.is_cuda and actions.dim() == 3
        state = state.contiguous().float()
        actions = actions.contiguous().float()
        B, delta, _ = actions.shape
        if out is None:
            out = torch.empty_like(state)
        if confidence is None:
            confidence = torch.empty((B,), dtype=torch.float32, device=state.device)
        jpi_corr_predict(self.handle, state, actions, B, delta, out, confidence, stream)
        return out, confidence

    def memory_usage(self) -> int:
        return jpi_corr_memory_usage(self.handle)
