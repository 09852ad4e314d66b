"""Builds the CUDA library libfastmtp.so in-tree (paper_2609_03181_gb300/_lib/) with nvcc for
sm_103a.  Translation units compile in parallel; the result is reused while the sources, the
header and the flags are unchanged.

The device-timeline variant (FM_TRACE defined: the per-CTA records read by spec_trace_read) is
the same sources built into paper_2609_03181_gb300/_lib_trace/.  build() returns the variant
that FASTMTP_TRACE=1 in the environment selects; build_all() compiles both."""
from __future__ import annotations

import hashlib
import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
TRACE = os.environ.get("FASTMTP_TRACE", "0") not in ("", "0")
SOURCES = ["gemm_tc.cu", "attention.cu", "small_kernels.cu", "runtime.cu", "noalloc.cu", "objective.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
BASE_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE]


def lib_dir(trace: bool) -> str:
    return os.path.join(PKG, "_lib_trace" if trace else "_lib")


def flags(trace: bool) -> list:
    return BASE_FLAGS + (["-DFM_TRACE"] if trace else [])


LIBDIR = lib_dir(TRACE)
LIB = os.path.join(LIBDIR, "libfastmtp.so")
FLAGS = flags(TRACE)


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the FastMTP CUDA library cannot be built")


def _digest(trace: bool) -> str:
    h = hashlib.sha256()
    for name in sorted(os.listdir(CSRC)):
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(name.encode() + f.read())
    with open(os.path.join(INCLUDE, "fastmtp.h"), "rb") as f:
        h.update(f.read())
    h.update(" ".join(ARCH + flags(trace)).encode())
    return h.hexdigest()


def _compile(jobs, verbose):
    """jobs: (source, object, flags); compiled in parallel."""
    nvcc = _nvcc()

    def one(job):
        src, obj, fl = job
        r = subprocess.run([nvcc, *ARCH, *fl, "-c", os.path.join(CSRC, src), "-o", obj], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose:
            print(r.stdout, r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 1)) as ex:
        return list(ex.map(one, jobs))


def _link(trace: bool, objs) -> str:
    d = lib_dir(trace)
    lib = os.path.join(d, "libfastmtp.so")
    tmp = lib + ".tmp"
    r = subprocess.run([_nvcc(), *ARCH, "-shared", "-o", tmp, *objs], capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    with open(os.path.join(d, "build.sha256"), "w") as f:
        f.write(_digest(trace))
    return lib


def _stale(trace: bool, force: bool) -> bool:
    d = lib_dir(trace)
    os.makedirs(d, exist_ok=True)
    stamp = os.path.join(d, "build.sha256")
    lib = os.path.join(d, "libfastmtp.so")
    return force or not (os.path.exists(lib) and os.path.exists(stamp) and open(stamp).read() == _digest(trace))


def build_all(force: bool = False, verbose: bool = False) -> list:
    """Compiles (if needed) the normal library and the device-timeline variant, all translation
    units of both in one parallel pool; returns the two library paths."""
    variants = [t for t in (False, True) if _stale(t, force)]
    jobs = [(src, os.path.join(lib_dir(t), src.replace(".cu", ".o")), flags(t)) for t in variants for src in SOURCES]
    objs = _compile(jobs, verbose) if jobs else []
    for k, t in enumerate(variants):
        _link(t, objs[k * len(SOURCES):(k + 1) * len(SOURCES)])
    return [os.path.join(lib_dir(t), "libfastmtp.so") for t in (False, True)]


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile (if needed) and return the path of the libfastmtp.so variant this process uses."""
    if _stale(TRACE, force):
        jobs = [(src, os.path.join(LIBDIR, src.replace(".cu", ".o")), FLAGS) for src in SOURCES]
        _link(TRACE, _compile(jobs, verbose))
    return LIB


if __name__ == "__main__":
    print(build_all(force=True, verbose=True))
