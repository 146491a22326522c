"""Builds libheadkv.so (the C-ABI of include/hkv.h) and the synthetic-input
generator library for sm_103a with nvcc, in tree.

Translation units compile in parallel; objects go to the package's _build/
folder, the shared libraries next to their Python wrappers.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libheadkv.so")
SYNTH_SRC = os.path.join(ROOT, "synth", "synth_gpu.cu")
SYNTH_LIB = os.path.join(ROOT, "synth", "libhkv_synth.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
         "-I", os.path.join(ROOT, "include"), "-I", CSRC]

SOURCES = ["hkv_api.cu", "hkv_attention.cu", "hkv_step.cu", "hkv_update.cu", "hkv_noalloc.cu"]


def nvcc() -> str:
    exe = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(exe):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libheadkv.so")
    return exe


def _run_all(cmds):
    procs = [(c, subprocess.Popen(c, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)) for c in cmds]
    errors = []
    for c, p in procs:
        out = p.communicate()[0].decode(errors="replace")
        if p.returncode != 0:
            errors.append(" ".join(c) + "\n" + out)
        elif out.strip() and os.environ.get("HKV_BUILD_VERBOSE"):
            sys.stderr.write(out)
    if errors:
        raise RuntimeError("nvcc failed:\n" + "\n".join(errors))


def _stale(target, deps):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, extra_flags=(), lib_path: str | None = None,
          build_dir: str | None = None) -> None:
    """Compiles the sources into lib_path (default: the package's
    libheadkv.so, objects in _build/); extra_flags (e.g. -D tuning macros) go
    to every nvcc call of the library."""
    lib = lib_path or LIB
    bdir = build_dir or (BUILD if lib_path is None else os.path.join(os.path.dirname(lib), "_build"))
    os.makedirs(bdir, exist_ok=True)
    cc = nvcc()
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    headers.append(os.path.join(ROOT, "include", "hkv.h"))
    objs, cmds = [], []
    for src in SOURCES:
        s = os.path.join(CSRC, src)
        o = os.path.join(bdir, src.replace(".cu", ".o"))
        objs.append(o)
        if force or _stale(o, [s] + headers):
            cmds.append([cc, *ARCH, *FLAGS, *extra_flags, "-c", s, "-o", o])
    synth_cmd = None
    if lib_path is None and (force or _stale(SYNTH_LIB, [SYNTH_SRC])):
        synth_cmd = [cc, *ARCH, "-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-shared",
                     SYNTH_SRC, "-o", SYNTH_LIB]
    _run_all(cmds + ([synth_cmd] if synth_cmd else []))
    if force or cmds or _stale(lib, objs):
        _run_all([[cc, *ARCH, "-shared", *objs, "-o", lib]])


if __name__ == "__main__":
    build(force="--force" in sys.argv)
    print(LIB)
