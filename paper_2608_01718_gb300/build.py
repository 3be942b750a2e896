"""Build liblacache.so in-tree for sm_103a (nvcc, one process per translation unit, then a shared link).

    python -m paper_2608_01718_gb300.build [-v]

Output: paper_2608_01718_gb300/_build/liblacache.so, and libpeaks.so (the benchmark's measurement kernels, not part
of the lookup library), both git-ignored. No cmake; nvcc and a C++ host compiler only.
"""
from __future__ import annotations

import fcntl
import os
import shutil
import subprocess
import sys
import tempfile

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "liblacache.so")
PEAKS_LIB = os.path.join(BUILD, "libpeaks.so")
PEAKS_SOURCE = "peaks.cu"

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
SOURCES = ["api.cu", "stage1_stream.cu", "stage1_tensor.cu", "stage2.cu", "noalloc.cu", "calibrate.cu", "lsh.cu",
           "lsh_tc.cu", "speculative.cu", "shards.cu"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build liblacache.so")


def flags(verbose: bool = False) -> list[str]:
    f = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC,
                "--expt-relaxed-constexpr"]
    if verbose:
        f += ["-Xptxas", "-v"]
    return f


def build(verbose: bool = False, force: bool = False) -> str:
    """Compile every CUDA source and link liblacache.so; returns its path. Concurrent callers (the ranks of a
    multi-GPU run, parallel test workers) take a file lock, so one of them compiles and the others then find the
    library up to date."""
    os.makedirs(BUILD, exist_ok=True)
    with open(os.path.join(BUILD, ".lock"), "w") as lock:
        fcntl.flock(lock, fcntl.LOCK_EX)
        try:
            return _build_locked(verbose, force)
        finally:
            fcntl.flock(lock, fcntl.LOCK_UN)


def _build_locked(verbose: bool, force: bool) -> str:
    srcs = [os.path.join(CSRC, s) for s in SOURCES]
    deps = srcs + [os.path.join(CSRC, h) for h in ("internal.cuh", "tcgen05.cuh")]
    deps += [os.path.join(INCLUDE, "lacache.h"), __file__]
    peaks_src = os.path.join(CSRC, PEAKS_SOURCE)
    lib_ok = os.path.exists(LIB) and os.path.getmtime(LIB) >= max(os.path.getmtime(p) for p in deps)
    peaks_ok = os.path.exists(PEAKS_LIB) and os.path.getmtime(PEAKS_LIB) >= max(os.path.getmtime(peaks_src),
                                                                                   os.path.getmtime(__file__))
    if not force and lib_ok and peaks_ok:
        return LIB
    tool = nvcc()
    objs, procs = [], []
    fd, peaks_tmp = tempfile.mkstemp(suffix=".so", dir=BUILD)
    os.close(fd)
    peaks = subprocess.Popen([tool, *flags(verbose), "-shared", peaks_src, "-o", peaks_tmp], stdout=subprocess.PIPE,
                             stderr=subprocess.STDOUT, text=True)
    for src in srcs:
        obj = os.path.join(BUILD, os.path.basename(src).replace(".cu", ".o"))
        objs.append(obj)
        cmd = [tool, *flags(verbose), "-c", src, "-o", obj]
        procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
    failed = []
    for src, proc in procs + [(peaks_src, peaks)]:
        out, _ = proc.communicate()
        if verbose or proc.returncode:
            sys.stderr.write(out)
        if proc.returncode:
            failed.append(src)
    if failed:
        os.unlink(peaks_tmp)
        raise RuntimeError(f"nvcc failed for {failed}")
    os.replace(peaks_tmp, PEAKS_LIB)
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=BUILD)
    os.close(fd)
    link = [tool, *ARCH, "-shared", "-Xcompiler", "-fPIC", "-o", tmp, *objs]
    res = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if res.returncode:
        os.unlink(tmp)
        raise RuntimeError("link of liblacache.so failed:\n" + res.stdout)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, force=True))
