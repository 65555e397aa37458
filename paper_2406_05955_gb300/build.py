"""Build libtsffn.so (the sm_103a CUDA kernels + C ABI) in-tree with nvcc.

Each translation unit compiles in parallel to an object with
``-gencode arch=compute_103a,code=sm_103a``; the objects link into
``paper_2406_05955_gb300/_build/libtsffn.so`` (CUDA runtime linked statically,
so the library needs only the driver at run time).
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
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(OUT_DIR, "libtsffn.so")
# The same sources with -DTS_DEBUG: every gathered row index is range-checked
# into the status word (see debug_row in csrc/ts_kernels.cuh).
DEBUG_DIR = os.path.join(OUT_DIR, "debug")
DEBUG_LIB = os.path.join(DEBUG_DIR, "libtsffn_debug.so")
SOURCES = ["ts_api.cu", "ts_gate_up.cu", "ts_down.cu", "ts_router.cu", "ts_noalloc.cu", "ts_wide.cu",
           "ts_topk.cu", "ts_predict.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libtsffn")


def _inputs() -> list[str]:
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cu", ".cuh", ".h"))]
    files += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h")]
    return files + [os.path.abspath(__file__)]


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def _build_libs(targets: list[tuple[str, str, list[str]]], verbose: bool) -> None:
    """Compile every (library, object dir, extra flags) target's sources in one pool, then link each."""
    cc = nvcc()
    jobs = []
    for lib, odir, flags in targets:
        os.makedirs(odir, exist_ok=True)
        jobs += [(src, odir, flags) for src in SOURCES]

    def compile_one(job) -> str:
        src, odir, flags = job
        obj = os.path.join(odir, src.replace(".cu", ".o"))
        cmd = [cc, *ARCH, *NVCC_FLAGS, *flags, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src} ({' '.join(flags)}):\n{r.stderr}")
        if verbose and r.stderr:
            sys.stderr.write(r.stderr)
        return obj

    with cf.ThreadPoolExecutor(max_workers=min(len(jobs), max(os.cpu_count() or 1, len(SOURCES)))) as ex:
        objs = list(ex.map(compile_one, jobs))
    for k, (lib, _, _) in enumerate(targets):
        tmp = lib + f".tmp{os.getpid()}"
        mine = objs[k * len(SOURCES):(k + 1) * len(SOURCES)]
        r = subprocess.run([cc, *ARCH, "-shared", "-o", tmp, *mine], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc link failed:\n{r.stderr}")
        os.replace(tmp, lib)


def build(force: bool = False, verbose: bool = False, extra: list[str] | None = None,
          debug: bool = True) -> str:
    """Compile and link libtsffn.so (and, with ``debug``, the range-checked
    libtsffn_debug.so) if any input changed; return the release library's path."""
    targets = []
    if force or not up_to_date(LIB):
        targets.append((LIB, OUT_DIR, list(extra or [])))
    if debug and (force or not up_to_date(DEBUG_LIB)):
        targets.append((DEBUG_LIB, DEBUG_DIR, ["-DTS_DEBUG", *(extra or [])]))
    if targets:
        _build_libs(targets, verbose)
    return LIB


if __name__ == "__main__":
    v = "-v" in sys.argv
    print(build(force=True, verbose=v, extra=["-Xptxas", "-v"] if v else None))
