"""Builds libriftgb.so (the C ABI of include/rift.h) in-tree with nvcc for sm_103a.

Each .cu file compiles in its own nvcc process (in parallel), then one link step.  Usage:
``python -m paper_2609_29029_gb300.build`` or ``build()`` from Python.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys
from pathlib import Path

PKG = Path(__file__).resolve().parent
ROOT = PKG.parent
CSRC = PKG / "csrc"
OBJ = PKG / "_build"
LIB = PKG / "libriftgb.so"
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and Path(cand).exists():
            return cand
    raise RuntimeError("nvcc not found: the Rift CUDA library cannot be built")


def sources() -> list:
    return sorted(CSRC.glob("*.cu"))


def _flags() -> list:
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
                   "-I", str(ROOT / "include"), "-I", str(CSRC)]


def _compile(src: Path, verbose_ptxas: bool) -> tuple:
    obj = OBJ / (src.stem + ".o")
    cmd = [nvcc()] + _flags() + (["-Xptxas", "-v"] if verbose_ptxas else []) + ["-c", str(src), "-o", str(obj)]
    p = subprocess.run(cmd, capture_output=True, text=True)
    return src, obj, p.returncode, p.stdout + p.stderr


def _stale(srcs) -> bool:
    if not LIB.exists():
        return True
    t = LIB.stat().st_mtime
    deps = list(srcs) + list(CSRC.glob("*.h")) + list(CSRC.glob("*.cuh")) + [ROOT / "include" / "rift.h", Path(__file__)]
    return any(p.stat().st_mtime > t for p in deps)


def build(force: bool = False, verbose_ptxas: bool = False, quiet: bool = True) -> Path:
    srcs = sources()
    if not force and not verbose_ptxas and not _stale(srcs):
        return LIB
    OBJ.mkdir(exist_ok=True)
    with cf.ThreadPoolExecutor(max_workers=min(len(srcs), os.cpu_count() or 4)) as ex:
        results = list(ex.map(lambda s: _compile(s, verbose_ptxas), srcs))
    failed = [r for r in results if r[2] != 0]
    for src, _, rc, out in results:
        if (rc != 0 or verbose_ptxas or not quiet) and out.strip():
            print(f"== {src.name}\n{out}", file=sys.stderr)
    if failed:
        raise RuntimeError("nvcc failed for: " + ", ".join(r[0].name for r in failed))
    tmp = LIB.with_suffix(".so.tmp")
    cmd = [nvcc()] + ARCH + ["-shared", "-cudart", "shared", "-o", str(tmp)] + [str(r[1]) for r in results] + [
        "-Xlinker", "-rpath,/usr/local/cuda/lib64"]
    p = subprocess.run(cmd, capture_output=True, text=True)
    if p.returncode != 0:
        raise RuntimeError("link failed:\n" + p.stdout + p.stderr)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose_ptxas="-v" in sys.argv, quiet=False)
    print(LIB)
