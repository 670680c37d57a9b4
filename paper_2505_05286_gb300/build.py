"""Builds the CUDA library libhxsim.so in-tree for sm_103a (GB300).

    python -m paper_2505_05286_gb300.build
"""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(PKG, "libhxsim.so")
# the bounds-checked build (-DHX_CHECKED): every index the simulation kernel
# forms is range-checked, a failure is a per-simulation status (HX_ERR_BOUNDS)
LIB_CHECKED = os.path.join(PKG, "libhxsim_checked.so")
SOURCES = ["hx_kernels.cu", "hx_api.cu"]
NVCC = os.environ.get("NVCC", "nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC]


def _stale(out: str) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(INCLUDE, "hxsim.h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False, extra=(), out: str = LIB, checked: bool = True) -> str:
    """Build `out` (default: libhxsim.so) and, with `checked`, the
    bounds-checked libhxsim_checked.so beside it, in parallel."""
    if out == LIB and checked:
        with ThreadPoolExecutor(2) as ex:
            jobs = [ex.submit(build, force, verbose, extra, LIB, False),
                    ex.submit(build, force, verbose, tuple(extra) + ("-DHX_CHECKED",), LIB_CHECKED, False)]
            return [j.result() for j in jobs][0]
    if not force and out in (LIB, LIB_CHECKED) and not _stale(out):
        return out
    objdir = os.path.join(os.path.dirname(out), "_build" + ("" if out == LIB else "_" + os.path.splitext(os.path.basename(out))[0]))
    os.makedirs(objdir, exist_ok=True)

    def compile_one(src):
        obj = os.path.join(objdir, src.replace(".cu", ".o"))
        cmd = [NVCC, *ARCH, *FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with ThreadPoolExecutor(len(SOURCES)) as ex:
        outs = list(ex.map(compile_one, SOURCES))
    if verbose:
        for _, err in outs:
            sys.stderr.write(err)
    tmp = out + f".tmp{os.getpid()}"
    cmd = [NVCC, *ARCH, "-shared", "-o", tmp] + [o for o, _ in outs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force=True, verbose="-v" in sys.argv))
