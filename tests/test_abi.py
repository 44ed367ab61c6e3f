"""Host-side checks of the C-ABI library that need no GPU: it builds, loads without a driver,
exports every entry point include/jpi.h declares, and rejects bad arguments before touching
the device."""

import ctypes
import subprocess

import pytest

from paper_2607_12659_gb300 import build, jpi


@pytest.fixture(scope="module")
def lib():
    build.build()
    return jpi.load()


def test_every_declared_entry_point_is_exported(lib):
    names = jpi.header_symbols()
    assert len(names) >= 11
    out = subprocess.run(["nm", "-D", "--defined-only", jpi.LIB_PATH], capture_output=True, text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    for n in names:
        assert n in exported, n
        assert hasattr(lib, n)
    # Nothing but the C-ABI leaks out of the library.
    assert all(e.startswith("jpi_") for e in exported), sorted(e for e in exported if not e.startswith("jpi_"))


def test_library_does_not_link_the_driver(lib):
    out = subprocess.run(["ldd", jpi.LIB_PATH], capture_output=True, text=True).stdout
    assert "libcuda.so" not in out and "libtorch" not in out


def test_null_arguments_are_rejected_on_the_host(lib):
    h = ctypes.c_void_p()
    assert lib.jpi_expert_create(None, None, ctypes.byref(h)) == -1
    assert b"NULL" in lib.jpi_last_error()
    assert lib.jpi_expert_create(None, None, None) == -1
    assert lib.jpi_denoise(None, None, None, 1, 1, 1, None, None) == -1
    assert lib.jpi_set_prefix_kv(None, None, None, 1, 1, 0, None) == -1
    assert lib.jpi_set_correction(None, None, 1, 0, None) == -1
    assert lib.jpi_expert_destroy(None) == 0
    b = ctypes.c_longlong()
    assert lib.jpi_memory_usage(None, ctypes.byref(b)) == -1


def test_bad_configs_are_rejected_before_any_device_call(lib):
    from synth import TINY
    w = jpi.jpi_weights()
    bad = [dict(n_kv_heads=2), dict(time_dim=63), dict(head_dim=48), dict(max_batch=0),
           dict(max_steps=65), dict(precision=7), dict(n_layers=0)]
    for kw in bad:
        cfg = jpi.make_config(TINY, 1, 8, 4, 4)
        for k, v in kw.items():
            setattr(cfg, k, v)
        h = ctypes.c_void_p()
        st = lib.jpi_expert_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h))
        assert st in (-1, -7, -2), (kw, st)
        assert h.value is None


def test_correction_module_arguments_are_checked_on_the_host(lib):
    from paper_2607_12659_gb300 import corr
    from synth import PI05_CORRECTION
    lib = corr.load()
    h = ctypes.c_void_p()
    assert lib.jpi_corr_create(None, None, ctypes.byref(h)) == -1
    assert lib.jpi_corr_create(None, None, None) == -1
    assert lib.jpi_corr_destroy(None) == 0
    assert lib.jpi_corr_compress(None, None, 1, 1, 1, None, None) == -1
    assert lib.jpi_corr_predict(None, None, None, 1, 1, None, None, None) == -1
    b = ctypes.c_longlong()
    assert lib.jpi_corr_memory_usage(None, ctypes.byref(b)) == -1
    w = corr.jpi_corr_weights()
    bad = [dict(width=1000), dict(head_dim=48), dict(n_heads=3), dict(n_items=0), dict(n_items=9),
           dict(max_delta=0), dict(max_delta=65), dict(n_joint=9), dict(max_batch=0), dict(precision=5),
           dict(n_heads=16, head_dim=64, n_items=8), dict(max_vlm_tokens=0), dict(d_vlm=0)]
    for kw in bad:
        cfg = corr.make_corr_config(PI05_CORRECTION, 1, 816)
        for k, v in kw.items():
            setattr(cfg, k, v)
        st = lib.jpi_corr_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h))
        assert st in (-1, -7), (kw, st)
        assert h.value is None
    # A valid shape whose joint blocks are missing is refused before any device call.
    cfg = corr.make_corr_config(PI05_CORRECTION, 1, 816)
    assert lib.jpi_corr_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == -1
    assert b"jb" in lib.jpi_last_error()
