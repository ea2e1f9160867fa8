"""Builds the CUDA library libcrc.so in-tree for sm_103a with nvcc.

Each translation unit is compiled in parallel, then linked into a shared
library under ``paper_2609_04895_gb300/_build``.  No GPU is needed to build.
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD, "libcrc.so")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
UNITS = ["api.cu", "router.cu", "scan.cu", "scan_traced.cu", "synth.cu", "noalloc.cu", "fused.cu",
         "fused_n16.cu", "fused_n32.cu", "fused_n64.cu", "fused_n128.cu", "policy.cu",
         "policy_lru.cu", "policy_lfu.cu", "policy_lrfu.cu", "policy_spatio.cu", "loss.cu",
         "transfer.cu", "probe.cu"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _deps():
    return (glob.glob(os.path.join(CSRC, "*")) + glob.glob(os.path.join(INCLUDE, "*.h"))
            + [os.path.abspath(__file__)])


DEBUG_BUILD = os.path.join(BUILD, "debug")
DEBUG_LIB = os.path.join(DEBUG_BUILD, "libcrc.so")


def stale(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    return any(os.path.getmtime(f) > t for f in _deps())


def build(force: bool = False, verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    """Compile and link libcrc.so if any source changed; returns its path.

    debug=True builds the checking flavour (-DCRC_DEBUG: every index a kernel
    derives is checked against its array's bound before use, a failed check
    latches CRC_EDEVICE and skips the access) into _build/debug/libcrc.so; the
    product library is not touched."""
    out_dir = DEBUG_BUILD if debug else BUILD
    lib = DEBUG_LIB if debug else LIB
    if not force and not stale(lib):
        return lib
    os.makedirs(out_dir, exist_ok=True)
    cc = nvcc()
    flags = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                    "-I", INCLUDE, "--expt-relaxed-constexpr"] + list(extra_flags)
    if debug:
        flags.append("-DCRC_DEBUG")

    def compile_unit(u):
        obj = os.path.join(out_dir, u.replace(".cu", ".o"))
        cmd = [cc] + flags + ["-c", os.path.join(CSRC, u), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {u}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout, r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=len(UNITS)) as ex:
        objs = list(ex.map(compile_unit, UNITS))
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [cc] + ARCH + ["-shared", "-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    import sys
    print(build(force=True, verbose="-v" in sys.argv,
                extra_flags=["-Xptxas", "-v"] if "-v" in sys.argv else ()))
