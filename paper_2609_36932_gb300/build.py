"""Build libfastrl_grpo.so (the CUDA path) in-tree for sm_103a.

Each .cu file is compiled by nvcc in parallel, then linked with the static CUDA runtime (and no
other library) into paper_2609_36932_gb300/_build/libfastrl_grpo.so.  Nothing is installed
outside the tree.

build(checked=True) makes libfastrl_grpo_checked.so from the same sources with GRPO_CHECKED
defined: the kernels then test every index they compute before using it and report failures
through grpo_debug_checks (same ABI; objects under _build/checked).  build_all() makes both.
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
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libfastrl_grpo.so")
CHECKED_DIR = os.path.join(OUT_DIR, "checked")
LIB_CHECKED = os.path.join(OUT_DIR, "libfastrl_grpo_checked.so")
SOURCES = ["api.cu", "advantage.cu", "prune.cu", "compact.cu", "loss.cu", "gspo.cu", "reduce.cu",
           "lmhead.cu", "gemm.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _deps():
    d = [os.path.join(CSRC, s) for s in SOURCES]
    d += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    d.append(os.path.join(INCLUDE, "fastrl_grpo.h"))
    d.append(os.path.abspath(__file__))
    return d


def stale(checked: bool = False) -> bool:
    lib = LIB_CHECKED if checked else LIB
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    return any(os.path.getmtime(p) > t for p in _deps())


def build(force: bool = False, verbose: bool = False, extra_flags=(), checked: bool = False) -> str:
    """Compile the library (the checked build with checked=True) if missing or stale; return the
    .so path."""
    lib = LIB_CHECKED if checked else LIB
    out_dir = CHECKED_DIR if checked else OUT_DIR
    if not force and not stale(checked):
        return lib
    os.makedirs(out_dir, exist_ok=True)
    cc = nvcc()
    flags = [*NVCC_FLAGS, *(["-DGRPO_CHECKED=1"] if checked else []), *extra_flags]

    def compile_one(src):
        obj = os.path.join(out_dir, src.replace(".cu", ".o"))
        cmd = [cc, *ARCH, *flags, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        return src, obj, r

    objs = []
    with concurrent.futures.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        for src, obj, r in ex.map(compile_one, SOURCES):
            if r.returncode != 0 or verbose:
                sys.stderr.write(r.stdout + r.stderr)
            if r.returncode != 0:
                raise RuntimeError("nvcc failed on %s" % src)
            objs.append(obj)
    tmp = lib + ".tmp.%d" % os.getpid()
    r = subprocess.run([cc, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *objs],
                       capture_output=True, text=True)
    if r.returncode != 0:
        sys.stderr.write(r.stdout + r.stderr)
        raise RuntimeError("link failed")
    os.replace(tmp, lib)
    return lib


def build_all(force: bool = False) -> None:
    """Both libraries, compiled side by side."""
    with concurrent.futures.ThreadPoolExecutor(max_workers=2) as ex:
        for f in [ex.submit(build, force, False, (), c) for c in (False, True)]:
            f.result()


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                extra_flags=["-Xptxas", "-v"] if "--ptxas-v" in sys.argv else []))
