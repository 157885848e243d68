"""Build libposeidon.so in-tree for sm_103a with nvcc.

Each translation unit under csrc/ compiles to _build/<name>.o in parallel
(the makespan kernels are template-instantiated per stage count, so they are
spread over several units); the objects are linked into
paper_2609_06086_gb300/libposeidon.so next to this file.
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "libposeidon.so")
# measurement tooling (the INT32 rate probe), kept out of the library's ABI
PROBE_SRC = os.path.join(PKG, "probe", "int32_probe.cu")
PROBE_LIB = os.path.join(PKG, "libposeidon_probe.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC"]


def nvcc() -> str:
    exe = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(exe):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libposeidon")
    return exe


def _deps_mtime() -> float:
    files = (glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(CSRC, "*.h")) +
             [os.path.join(ROOT, "include", "poseidon.h")])
    return max(os.path.getmtime(f) for f in files)


def _compile(src: str, verbose: bool, force: bool) -> str:
    obj = os.path.join(BUILD, os.path.basename(src)[:-3] + ".o")
    if (not force and os.path.exists(obj) and
            os.path.getmtime(obj) >= max(os.path.getmtime(src), _deps_mtime())):
        return obj
    cmd = [nvcc(), *ARCH, *FLAGS, "-c", src, "-o", obj + ".tmp"]
    if verbose:
        cmd.insert(1, "-Xptxas=-v")
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    if verbose and r.stderr:
        sys.stderr.write(r.stderr)
    os.replace(obj + ".tmp", obj)
    return obj


def _build_probe(force: bool) -> str:
    hdr = os.path.join(ROOT, "include", "poseidon_probe.h")
    if (force or not os.path.exists(PROBE_LIB) or
            os.path.getmtime(PROBE_LIB) < max(os.path.getmtime(PROBE_SRC), os.path.getmtime(hdr))):
        tmp = PROBE_LIB + f".tmp{os.getpid()}"
        r = subprocess.run([nvcc(), *ARCH, *FLAGS, "-shared", PROBE_SRC, "-o", tmp],
                           capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {PROBE_SRC}:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, PROBE_LIB)
    return PROBE_LIB


def build(force: bool = False, verbose: bool = False, jobs: int | None = None) -> str:
    """Compile every csrc/*.cu and link libposeidon.so (and the measurement
    probe, libposeidon_probe.so); returns the library's path."""
    os.makedirs(BUILD, exist_ok=True)
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    jobs = jobs or max(1, min(len(srcs) + 1, os.cpu_count() or 1))
    # the heaviest units (many unrolled instantiations) first
    srcs.sort(key=lambda s: (0 if "range" in s or "leaf" in s else 1, s))
    with ThreadPoolExecutor(jobs) as ex:
        probe = ex.submit(_build_probe, force)
        objs = list(ex.map(lambda s: _compile(s, verbose, force), srcs))
        probe.result()
    if (force or not os.path.exists(LIB) or
            os.path.getmtime(LIB) < max(os.path.getmtime(o) for o in objs)):
        tmp = LIB + f".tmp{os.getpid()}"
        r = subprocess.run([nvcc(), *ARCH, "-shared", "-o", tmp, *sorted(objs)],
                           capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    import time
    t0 = time.time()
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv), f"{time.time() - t0:.1f}s")
