"""Host-side checks of the C-ABI libraries that need no GPU: they build, load without a driver,
export every entry point their headers declare (libjpi.so: include/jpi.h and jpi_corr.h;
libjpi_prefill.so: jpi_prefill.h), and reject bad arguments before touching the device."""

import ctypes
import os
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


def test_every_header_belongs_to_a_library():
    from paper_2607_12659_gb300 import prefill
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    headers = {f for f in os.listdir(inc) if f.endswith(".h")}
    assert headers == set(jpi.LIB_HEADERS) | {"jpi_prefill.h"}
    assert len(prefill.header_symbols()) == 6


def test_prefill_library_exports_its_entry_points_and_checks_arguments(lib):
    from paper_2607_12659_gb300 import build as b, prefill
    from synth import GEMMA2B
    assert b.PREFILL_BUILD_ERROR is None, b.PREFILL_BUILD_ERROR
    plib = prefill.load()
    out = subprocess.run(["nm", "-D", "--defined-only", prefill.LIB_PATH], capture_output=True, text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    assert exported == set(prefill.header_symbols())
    ldd = subprocess.run(["ldd", prefill.LIB_PATH], capture_output=True, text=True).stdout
    # Its products run on its own tensor-core kernel: no library GEMM, no driver or torch link.
    assert "libcublas" not in ldd and "libcuda.so" not in ldd and "libtorch" not in ldd
    h = ctypes.c_void_p()
    assert plib.jpi_prefill_create(None, None, ctypes.byref(h)) == -1
    assert b"NULL" in plib.jpi_prefill_last_error()
    assert plib.jpi_prefill_destroy(None) == 0
    assert plib.jpi_prefill_run(None, None, 1, 1, 1, None, None, 256, None, None) == -1
    n = ctypes.c_longlong()
    assert plib.jpi_prefill_memory_usage(None, ctypes.byref(n)) == -1
    assert plib.jpi_prefill_device_status(None) == -1
    w = prefill.jpi_prefill_weights()
    bad = [dict(n_layers=0), dict(width=2044), dict(head_dim=250), dict(head_dim=1024), dict(mlp_dim=12),
           dict(max_batch=0), dict(max_prefix=0), dict(rms_eps=-1.0), dict(max_prefix=70000)]
    for kw in bad:
        cfg = prefill.make_prefill_config(GEMMA2B, 1, 816)
        for k, v in kw.items():
            setattr(cfg, k, v)
        st = plib.jpi_prefill_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h))
        assert st in (-1, -7), (kw, st)
        assert h.value is None
    cfg = prefill.make_prefill_config(GEMMA2B, 1, 816)
    assert plib.jpi_prefill_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == -1   # NULL weights
    assert b"NULL" in plib.jpi_prefill_last_error()


def test_prefill_into_expert_refuses_stores_it_does_not_fit():
    # The C-ABI cannot see the size of the destination store; the binding checks it first.
    from types import SimpleNamespace as NS
    from paper_2607_12659_gb300.prefill import Prefill
    me = NS(dims=NS(n_layers=2, head_dim=128))
    store = dict(max_batch=2, max_prefix=64, n_layers=2, head_dim=128)
    for x_shape, dims, cfg in [((3, 40, 256), dict(precision="bf16"), store),
                               ((1, 65, 256), dict(precision="bf16"), store),
                               ((1, 40, 256), dict(precision="fp32"), store),
                               ((1, 40, 256), dict(precision="bf16"), {**store, "n_layers": 3}),
                               ((1, 40, 256), dict(precision="bf16"), {**store, "head_dim": 64})]:
        with pytest.raises(ValueError):
            Prefill.into_expert(me, NS(shape=x_shape), NS(dims=NS(**dims), cfg=NS(**cfg)))


def _c_layout(struct, fields, tmp_path):
    """sizeof and offsetof of a C struct from the public headers, by compiling a probe with gcc."""
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    src = tmp_path / f"{struct}.c"
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "jpi.h"', '#include "jpi_corr.h"',
             '#include "jpi_prefill.h"', "int main(void) {", f'  printf("%zu\\n", sizeof({struct}));']
    lines += [f'  printf("%zu\\n", offsetof({struct}, {f}));' for f in fields]
    lines += ["  return 0;", "}"]
    src.write_text("\n".join(lines))
    exe = tmp_path / struct
    subprocess.run(["gcc", "-I", inc, str(src), "-o", str(exe)], check=True, capture_output=True)
    out = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    return out[0], out[1:]


@pytest.mark.parametrize("mod,name", [("jpi", "jpi_config"), ("jpi", "jpi_weights"), ("corr", "jpi_corr_config"),
                                      ("corr", "jpi_corr_block"), ("corr", "jpi_corr_weights"),
                                      ("prefill", "jpi_prefill_config"), ("prefill", "jpi_prefill_weights")])
def test_binding_structs_match_the_c_layout(mod, name, tmp_path):
    import importlib
    m = importlib.import_module(f"paper_2607_12659_gb300.{mod}")
    st = getattr(m, name)
    fields = [f[0] for f in st._fields_]
    size, offsets = _c_layout(name, fields, tmp_path)
    assert ctypes.sizeof(st) == size, (name, ctypes.sizeof(st), size)
    assert [getattr(st, f).offset for f in fields] == offsets, name


def _header_params():
    """Parameter kinds ('ptr', 'int', 'float', 'longlong') of every JPI_API function in include/*.h."""
    import re
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    sig = {}
    for f in os.listdir(inc):
        text = re.sub(r"/\*.*?\*/", "", open(os.path.join(inc, f)).read(), flags=re.S)
        for m in re.finditer(r"JPI_API\s+[\w\s\*]+?\b(jpi_\w+)\s*\(([^;]*?)\)\s*;", text, flags=re.S):
            params = m.group(2).strip()
            kinds = []
            for p in ([] if params in ("", "void") else params.split(",")):
                p = " ".join(p.split())
                if "*" in p:
                    kinds.append("ptr")
                elif p.startswith("long long"):
                    kinds.append("longlong")
                elif p.startswith("float"):
                    kinds.append("float")
                else:
                    assert p.startswith("int "), p
                    kinds.append("int")
            sig[m.group(1)] = kinds
    return sig


def test_binding_signatures_match_the_c_prototypes():
    from paper_2607_12659_gb300 import corr, prefill
    want = _header_params()
    sigs = {**jpi._SIGS, **corr._SIGS, **prefill._SIGS}
    assert set(sigs) | {"jpi_last_error", "jpi_prefill_last_error"} == set(want)

    def kind(t):
        if t is ctypes.c_void_p or hasattr(t, "_type_") and isinstance(t, type(ctypes.POINTER(ctypes.c_int))):
            return "ptr"
        return {ctypes.c_int: "int", ctypes.c_float: "float", ctypes.c_longlong: "longlong"}[t]

    for name, args in sigs.items():
        assert [kind(a) for a in args] == want[name], (name, [kind(a) for a in args], want[name])
