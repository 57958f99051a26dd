"""Build libkvm.so (the CUDA kernels and the C ABI) in-tree for sm_103a.

    python -m paper_2609_18935_gb300.build_lib

Each translation unit is compiled in parallel with nvcc, then linked into
paper_2609_18935_gb300/_build/libkvm.so with the CUDA runtime linked
statically, so loading the library needs only the driver.
"""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "libkvm.so")
SOURCES = ["kvm_api.cu", "kv_compact.cu", "tail_attn.cu", "tail_attn_tc.cu", "gdn_scan_tc.cu", "attn_probe.cu", "gdn_conv.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
         "--expt-relaxed-constexpr", "-cudart", "static"]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.sep not in cand or os.path.exists(cand)):
            return cand
    raise RuntimeError("nvcc not found")


def _run(cmd):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("command failed:\n" + " ".join(cmd) + "\n" + r.stdout + r.stderr)
    return r.stdout + r.stderr


DEBUG_LIB = os.path.join(BUILD, "debug", "libkvm_debug.so")


def build(verbose_ptxas: bool = False, force: bool = False, debug: bool = False) -> str:
    """Build libkvm.so, or with `debug` the canary-checking variant
    _build/debug/libkvm_debug.so (-DKVM_DEBUG: every device buffer of a
    context between two canary bands that kvm_check verifies)."""
    out_dir = os.path.dirname(DEBUG_LIB) if debug else BUILD
    lib = DEBUG_LIB if debug else LIB
    os.makedirs(out_dir, exist_ok=True)
    nvcc = _nvcc()
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + \
           [os.path.join(PKG, "..", "include", "kvm.h")]
    newest_src = max(os.path.getmtime(p) for p in deps)
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= newest_src:
        return lib
    extra = (["-Xptxas", "-v"] if verbose_ptxas else []) + (["-DKVM_DEBUG"] if debug else [])

    def compile_one(src):
        obj = os.path.join(out_dir, src.replace(".cu", ".o"))
        out = _run([nvcc, *ARCH, *FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj])
        return obj, out

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    logs = "".join(o for _, o in results)
    tmp = lib + ".tmp"
    _run([nvcc, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *[o for o, _ in results]])
    os.replace(tmp, lib)
    if verbose_ptxas:
        sys.stdout.write(logs)
    return lib


if __name__ == "__main__":
    print(build(verbose_ptxas="-v" in sys.argv, force=True))
