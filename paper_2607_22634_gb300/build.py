"""Compile the sm_103a CUDA sources into the in-tree shared libraries.

libpresto.so is the library; libpresto_checks.so is the same sources compiled with
-DPRESTO_CHECKS (device-side bounds checks that report PRESTO_DEV_BOUNDS instead of
faulting), loaded instead when the environment sets PRESTO_CHECKS=1.  Each
translation unit compiles in parallel with one -gencode (sm_103a), then nvcc links
them with the static CUDA runtime, so a library needs only the driver at run time.
Rebuilds only when a source or header is newer than the library.
"""

from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OBJDIR = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libpresto.so")
CHECKS_LIB = os.path.join(HERE, "libpresto_checks.so")
SOURCES = ["api.cu", "topk.cu", "tree_build.cu", "tree_mask_accept.cu", "tree_attention.cu",
           "tree_attention_pair.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                "--expt-relaxed-constexpr", "-I", INCLUDE, "-I", CSRC]


def checks_requested() -> bool:
    """True when the environment asks for the bounds-checked debug library."""
    return os.environ.get("PRESTO_CHECKS", "") == "1"


def lib_file(checks: bool | None = None) -> str:
    """The library this process loads: the debug build under PRESTO_CHECKS=1."""
    if checks is None:
        checks = checks_requested()
    return CHECKS_LIB if checks else LIB


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the PRESTO CUDA library cannot be built")


def _inputs():
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    deps += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    deps.append(os.path.abspath(__file__))
    return deps


def up_to_date(checks: bool | None = None) -> bool:
    lib = lib_file(checks)
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _inputs())


def _run(cmd):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("command failed: " + " ".join(cmd) + "\n" + r.stdout + r.stderr)
    return r.stdout + r.stderr


def build(force: bool = False, verbose: bool = False, extra_flags=(), checks=None) -> str:
    """Build a library (if stale) and return its path: the one this process loads
    (`checks` None), the release library (False), the debug library (True), or both
    ("both", compiled in one parallel pool; returns the release path)."""
    variants = [False, True] if checks == "both" else [checks_requested() if checks is None else checks]
    todo = [v for v in variants if force or not up_to_date(v)]
    cc = nvcc() if todo else None
    jobs = []
    for v in todo:
        objdir = OBJDIR + ("_checks" if v else "")
        os.makedirs(objdir, exist_ok=True)
        defs = ["-DPRESTO_CHECKS"] if v else []
        for src in SOURCES:
            obj = os.path.join(objdir, src.replace(".cu", ".o"))
            jobs.append((v, obj, [cc, *FLAGS, *defs, *extra_flags, "-c", os.path.join(CSRC, src), "-o", obj]))
    if jobs:
        with concurrent.futures.ThreadPoolExecutor(max_workers=len(jobs)) as ex:
            logs = list(ex.map(lambda j: _run(j[2]), jobs))
        if verbose:
            for log in logs:
                sys.stdout.write(log)
    for v in todo:
        lib = lib_file(v)
        tmp = lib + ".tmp"
        _run([cc, *ARCH, "-shared", "-o", tmp, *[j[1] for j in jobs if j[0] == v]])
        os.replace(tmp, lib)
    return lib_file(False if checks == "both" else variants[0])


if __name__ == "__main__":
    v = "-v" in sys.argv
    extra = ["-Xptxas", "-v"] if "--ptxas" in sys.argv else []
    print(build(force=True, verbose=v or bool(extra), extra_flags=extra))
