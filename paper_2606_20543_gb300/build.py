"""Build libssd.so in-tree: every .cu under csrc/ compiled for sm_103a in
parallel with nvcc, linked with the static CUDA runtime (the library then
needs only the driver at run time).  Usage: python -m paper_2606_20543_gb300.build
[--force] [-v] [--debug-bounds]; --debug-bounds builds libssd_debug.so with
SSD_DEBUG_BOUNDS=1 (the kernels' index checks, recorded in the status word),
which the binding loads when SSD_LIBRARY=debug is set.
"""
from __future__ import annotations

import hashlib
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libssd.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
         "-I" + os.path.join(ROOT, "include")]
# Extra nvcc flags (for example -DSSD_ACCEPT_RSTAGES=8 to retune a kernel).
FLAGS += os.environ.get("SSD_NVCC_EXTRA", "").split()


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: libssd needs the CUDA 13 toolkit to build")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


DEBUG_BUILD = os.path.join(HERE, "_build_debug")
DEBUG_LIB = os.path.join(HERE, "libssd_debug.so")
DEBUG_FLAGS = ["-DSSD_DEBUG_BOUNDS=1"]


def _digest(flags=None) -> str:
    flags = FLAGS if flags is None else flags
    h = hashlib.sha256()
    for p in sorted(os.listdir(CSRC)) + ["../../include/ssd.h"]:
        path = os.path.normpath(os.path.join(CSRC, p))
        if os.path.isfile(path):
            h.update(p.encode())
            h.update(open(path, "rb").read())
    h.update(" ".join(ARCH + flags).encode())
    h.update(os.uname().machine.encode())
    return h.hexdigest()


def build(force: bool = False, verbose: bool = False, debug_bounds: bool = False) -> str:
    """Compile (if sources changed) and return the path of libssd.so (or,
    with debug_bounds, of libssd_debug.so)."""
    build_dir, lib = (DEBUG_BUILD, DEBUG_LIB) if debug_bounds else (BUILD, LIB)
    flags = FLAGS + (DEBUG_FLAGS if debug_bounds else [])
    os.makedirs(build_dir, exist_ok=True)
    stamp = os.path.join(build_dir, "stamp")
    dig = _digest(flags)
    if not force and os.path.exists(lib) and os.path.exists(stamp) and open(stamp).read() == dig:
        return lib
    cc = nvcc()
    procs = []
    objs = []
    for src in sources():
        obj = os.path.join(build_dir, os.path.basename(src)[:-3] + ".o")
        objs.append(obj)
        cmd = [cc] + ARCH + flags + ["-c", src, "-o", obj]
        if verbose:
            cmd += ["-Xptxas", "-v"]
        procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)))
    failed = []
    for src, p in procs:
        out = p.communicate()[0].decode()
        if p.returncode != 0:
            failed.append(f"{src}:\n{out}")
        elif verbose and out.strip():
            print(out)
    if failed:
        raise RuntimeError("nvcc failed:\n" + "\n".join(failed))
    tmp = lib + ".tmp"
    link = [cc] + ARCH + ["-shared", "-o", tmp] + objs + ["-cudart", "static"]
    r = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n" + r.stdout.decode())
    os.replace(tmp, lib)
    with open(stamp, "w") as f:
        f.write(dig)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                debug_bounds="--debug-bounds" in sys.argv))
