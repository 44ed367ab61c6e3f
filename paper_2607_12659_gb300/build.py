"""Builds the libraries in-tree for sm_103a with nvcc (no cmake, no torch build).

``libjpi.so``: the action expert and the future correction module (every .cu directly under
csrc/). Each translation unit compiles in parallel; the objects link into one shared library
with the CUDA runtime linked statically, so the library needs no libcuda at load time (the
driver entry points are resolved at run time).

``libjpi_prefill.so``: the LLM prefill (csrc/prefill/), its own tensor-core kernels, linked the
same way. A failure to build it leaves only the prefill unbuilt (reported on stderr and by
``PREFILL_BUILD_ERROR``).
"""

from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libjpi.so")
PREFILL_SRC = os.path.join(CSRC, "prefill")
PREFILL_LIB = os.path.join(PKG, "libjpi_prefill.so")
PREFILL_BUILD_ERROR = None

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + [
    "-O3", "-lineinfo", "-std=c++17", "--expt-relaxed-constexpr",
    "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
    "-I", os.path.join(ROOT, "include"),
]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libjpi.so")


def sources() -> list[str]:
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _stale(obj: str, src: str) -> bool:
    if not os.path.exists(obj):
        return True
    t = os.path.getmtime(obj)
    inc = os.path.join(ROOT, "include")
    deps = [src] + [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    deps += [os.path.join(inc, f) for f in os.listdir(inc) if f.endswith(".h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build_prefill(verbose: bool = False, force: bool = False) -> str:
    """Compile csrc/prefill/*.cu and link libjpi_prefill.so."""
    cc = nvcc()
    out = os.path.join(BUILD, "prefill")
    os.makedirs(out, exist_ok=True)
    srcs = sorted(os.path.join(PREFILL_SRC, f) for f in os.listdir(PREFILL_SRC) if f.endswith(".cu"))
    headers = [os.path.join(ROOT, "include", f) for f in ("jpi.h", "jpi_prefill.h")] + [
        os.path.join(CSRC, f) for f in ("ptx.h", "attn_t5_kernel.cuh")]
    objs = []
    for src in srcs:
        obj = os.path.join(out, os.path.basename(src)[:-3] + ".o")
        objs.append(obj)
        if not force and os.path.exists(obj) and all(
                os.path.getmtime(d) <= os.path.getmtime(obj) for d in [src] + headers):
            continue
        r = subprocess.run([cc] + NVCC_FLAGS + ["-c", src, "-o", obj], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {os.path.basename(src)}:\n{r.stderr}")
        if verbose and r.stderr:
            print(r.stderr, file=sys.stderr)
    if force or not os.path.exists(PREFILL_LIB) or any(
            os.path.getmtime(o) > os.path.getmtime(PREFILL_LIB) for o in objs):
        tmp = PREFILL_LIB + ".tmp"
        cmd = [cc] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link of libjpi_prefill.so failed:\n{r.stderr}")
        os.replace(tmp, PREFILL_LIB)
    return PREFILL_LIB


PROBE_SRC = os.path.join(CSRC, "probe", "primitives.cu")
PROBE_BIN = os.path.join(BUILD, "primitives")


def build_probe(force: bool = False) -> str:
    """Compile the hardware-primitive diagnostic (csrc/probe/primitives.cu, a standalone
    executable, not part of either library) and return its path."""
    os.makedirs(BUILD, exist_ok=True)
    deps = [PROBE_SRC, os.path.join(CSRC, "ptx.h")]
    if force or not os.path.exists(PROBE_BIN) or any(os.path.getmtime(d) > os.path.getmtime(PROBE_BIN) for d in deps):
        r = subprocess.run([nvcc()] + ARCH + ["-O2", "-std=c++17", "-o", PROBE_BIN, PROBE_SRC],
                           capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for primitives.cu:\n{r.stderr}")
    return PROBE_BIN


def build(verbose: bool = False, force: bool = False) -> str:
    """Compile every .cu directly under csrc/ and link libjpi.so, then the prefill library;
    returns libjpi.so's path."""
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    srcs = sources()
    objs = [os.path.join(BUILD, os.path.basename(s)[:-3] + ".o") for s in srcs]

    def compile_one(pair):
        src, obj = pair
        if not force and not _stale(obj, src):
            return None
        cmd = [cc] + NVCC_FLAGS + ["-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {os.path.basename(src)}:\n{r.stderr}")
        return r.stderr if verbose else None

    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(srcs), os.cpu_count() or 4))) as ex:
        for msg in ex.map(compile_one, zip(srcs, objs)):
            if msg:
                print(msg, file=sys.stderr)
    relink = force or not os.path.exists(LIB) or any(
        os.path.getmtime(o) > os.path.getmtime(LIB) for o in objs)
    if relink:
        tmp = LIB + ".tmp"
        cmd = [cc] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stderr}")
        os.replace(tmp, LIB)
    global PREFILL_BUILD_ERROR
    try:
        build_prefill(verbose, force)
        PREFILL_BUILD_ERROR = None
    except (RuntimeError, OSError) as e:
        PREFILL_BUILD_ERROR = str(e)
        print(f"warning: libjpi_prefill.so not built: {e}", file=sys.stderr)
    return LIB


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, force="-f" in sys.argv))
