"""Builds libsolo_readout.so in-tree with nvcc for sm_103a.

The translation units compile in parallel; the shared library links
the CUDA runtime statically, so loading it needs no GPU and no libcuda
(the driver is reached through the runtime's entry-point query at the
first call).
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
LIBDIR = os.path.join(HERE, "lib")
LIB = os.path.join(LIBDIR, "libsolo_readout.so")
# The checked build: every computed global index of the row kernels and GEMM
# epilogues is tested (SOLO_DEBUG=1); a violation sets SOLO_FLAG_BOUNDS.
LIB_CHECKED = os.path.join(LIBDIR, "libsolo_readout_checked.so")
SOURCES = ["gemm_tc.cu", "rowops.cu", "solo_readout.cu", "selftest.cu", "flash_bwd.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build libsolo_readout")


def _inputs() -> list[str]:
    files = [os.path.join(CSRC, s) for s in SOURCES]
    files += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    files.append(os.path.join(os.path.dirname(HERE), "include", "solo_readout.h"))
    return files


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def up_to_date_checked() -> bool:
    return up_to_date(LIB_CHECKED)


def build(verbose: bool = False, extra_flags: list[str] | None = None,
          checked: bool = False) -> str:
    """Compiles the release library (or, with checked=True, the checked one)."""
    os.makedirs(LIBDIR, exist_ok=True)
    cc = nvcc()
    extra = list(extra_flags or []) + (["-DSOLO_DEBUG=1"] if checked else [])
    target = LIB_CHECKED if checked else LIB
    tag = "_checked" if checked else ""
    objs, procs = [], []
    for src in SOURCES:
        obj = os.path.join(LIBDIR, src.replace(".cu", tag + ".o"))
        cmd = [cc, *ARCH, *FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)))
        objs.append(obj)
    failed = []
    for src, p in procs:
        out, _ = p.communicate()
        if verbose or p.returncode:
            sys.stdout.write(out.decode(errors="replace"))
        if p.returncode:
            failed.append(src)
    if failed:
        raise RuntimeError(f"nvcc failed on {failed}")
    tmp = target + ".tmp"
    cmd = [cc, *ARCH, "-shared", *objs, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, target)
    for o in objs:
        os.remove(o)
    return target


def build_all(verbose: bool = False) -> list[str]:
    """The release and the checked library, compiled concurrently."""
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(2) as ex:
        futs = [ex.submit(build, verbose, None, c) for c in (False, True)]
        return [f.result() for f in futs]


def ensure_built() -> str:
    if not up_to_date():
        build()
    return LIB


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv,
                extra_flags=["-Xptxas", "-v"] if "--ptxas" in sys.argv else None))
