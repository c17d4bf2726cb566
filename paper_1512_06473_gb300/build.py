"""Build libqcnn.so (the CUDA kernels and the C ABI of include/qcnn.h) for
sm_103a with nvcc, in-tree under paper_1512_06473_gb300/_build/.

Each .cu file is compiled in parallel, then linked into one shared library
with the CUDA runtime linked statically (the library only needs the driver).
The same sources also build libqcnn_debug.so under _build_debug/, with the
kernels' device checks compiled in (QCNN_DEBUG_CHECKS).
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD, "libqcnn.so")
# Debug build: every kernel also records codes >= K and out-of-range indices
# (QCNN_DEBUG_CHECKS; read back by qcnn_device_check).  Same sources, same ABI.
BUILD_DEBUG = os.path.join(HERE, "_build_debug")
LIB_DEBUG = os.path.join(BUILD_DEBUG, "libqcnn_debug.so")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-I", INCLUDE]
DEBUG_FLAGS = ["-DQCNN_DEBUG_CHECKS"]


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libqcnn")


def sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return sources() + sorted(glob.glob(os.path.join(CSRC, "*.cuh"))) + [os.path.join(INCLUDE, "qcnn.h")]


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _deps())


def _variants(debug: bool):
    v = [(BUILD, LIB, [])]
    if debug:
        v.append((BUILD_DEBUG, LIB_DEBUG, DEBUG_FLAGS))
    return v


def build(force: bool = False, verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    """Compile every .cu under csrc/ for sm_103a and link libqcnn.so; with
    debug=True also libqcnn_debug.so (all translation units of both compiled
    in one parallel pool).  Returns the release library's path."""
    todo = [(d, lib, fl) for d, lib, fl in _variants(debug) if force or not up_to_date(lib)]
    if not todo:
        return LIB
    cc = nvcc()
    jobs = []
    for d, lib, fl in todo:
        os.makedirs(d, exist_ok=True)
        for src in sources():
            jobs.append((d, fl, src))

    def compile_one(job):
        d, fl, src = job
        obj = os.path.join(d, os.path.basename(src)[:-3] + ".o")
        cmd = [cc, *ARCH, *NVCC_FLAGS, *fl, *extra_flags, "-c", src, "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    # the largest translation units first, so they do not finish last
    jobs.sort(key=lambda j: -os.path.getsize(j[2]))
    objs = {d: [] for d, _, _ in todo}
    with cf.ThreadPoolExecutor(max_workers=min(32, os.cpu_count() or 1)) as ex:
        for job, (obj, log) in zip(jobs, ex.map(compile_one, jobs)):
            objs[job[0]].append(obj)
            if verbose and log:
                sys.stderr.write(log)
    for d, lib, _ in todo:
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [cc, *ARCH, "-shared", "-Xlinker", "-Bsymbolic", "-o", tmp, *sorted(objs[d])]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return LIB


def build_debug(force: bool = False) -> str:
    """Build (when stale) and return the debug library libqcnn_debug.so."""
    if force or not up_to_date(LIB_DEBUG):
        build(force=force, debug=True)
    return LIB_DEBUG


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                debug="--debug" in sys.argv))
