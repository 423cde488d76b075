"""Build libtac.so in-tree for sm_103a.

Every kernel instance (d x dtype) is its own nvcc invocation of the same source
file, run in parallel, then everything is linked into ``_build/libtac.so``.
A stamp of the sources, flags and nvcc version skips rebuilding when nothing
changed.  No CMake, no torch extension machinery.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
OUT = os.path.join(HERE, "_build")
LIB = os.path.join(OUT, "libtac.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CFLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fno-strict-aliasing",
          "--expt-relaxed-constexpr"]


def _units():
    units = [("tac_api.cu", [], "tac_api"), ("tac_fwht_debug.cu", [], "tac_fwht_debug"),
             ("tac_attend.cu", [], "tac_attend")]
    for kind in ("encode", "decode"):
        for t in ("BF16", "F32"):
            for d in (128, 64, 32, 16):  # biggest first: they dominate the wall time
                units.append((f"tac_{kind}.cu", [f"-DTAC_INST_D={d}", f"-DTAC_INST_{t}=1"],
                              f"tac_{kind}_{d}_{t.lower()}"))
    return units


def _nvcc() -> str:
    p = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(p):
        raise RuntimeError("nvcc not found: libtac needs the CUDA toolkit to build")
    return p


def _stamp(nvcc: str) -> str:
    h = hashlib.sha256()
    for root in (CSRC, INCLUDE):
        for name in sorted(os.listdir(root)):
            if name.endswith((".cu", ".cuh", ".h")):
                with open(os.path.join(root, name), "rb") as f:
                    h.update(name.encode() + b"\0" + f.read())
    h.update(" ".join(ARCH + CFLAGS).encode())
    try:
        h.update(subprocess.run([nvcc, "--version"], capture_output=True, text=True).stdout.encode())
    except OSError:
        pass
    return h.hexdigest()


def build(force: bool = False, jobs: int | None = None, verbose: bool = False) -> str:
    """Compile and link libtac.so if needed; returns its path."""
    nvcc = _nvcc()
    os.makedirs(os.path.join(OUT, "obj"), exist_ok=True)
    stamp = _stamp(nvcc)
    stamp_file = os.path.join(OUT, "stamp")
    if not force and os.path.exists(LIB) and os.path.exists(stamp_file):
        with open(stamp_file) as f:
            if f.read().strip() == stamp:
                return LIB

    def compile_one(unit):
        src, defs, name = unit
        obj = os.path.join(OUT, "obj", name + ".o")
        cmd = [nvcc] + ARCH + CFLAGS + defs + ["-I", INCLUDE, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {name}:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        if verbose:
            sys.stderr.write(f"[libtac] built {name}\n")
        return obj

    units = _units()
    workers = jobs or min(len(units), max(1, os.cpu_count() or 1))
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        objs = list(ex.map(compile_one, units))
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [nvcc] + ARCH + ["-shared", "-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(stamp_file, "w") as f:
        f.write(stamp)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
