"""Builds libgroupsparse.so (the C-ABI library) in-tree with nvcc for sm_103a.

Each translation unit is compiled in parallel to an object under
`paper_2609_33977_gb300/_build/`, then linked into
`paper_2609_33977_gb300/libgroupsparse.so` against the shared CUDA runtime.
A rebuild happens only when a source or header is newer than the library.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys
from pathlib import Path

PKG = Path(__file__).resolve().parent
CSRC = PKG / "csrc"
INCLUDE = PKG.parent / "include"
BUILD = PKG / "_build"
LIB = PKG / "libgroupsparse.so"
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _nvcc() -> str:
    for cand in (os.environ.get("CUDA_HOME", ""), "/usr/local/cuda"):
        if cand and (Path(cand) / "bin" / "nvcc").exists():
            return str(Path(cand) / "bin" / "nvcc")
    found = shutil.which("nvcc")
    if not found:
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libgroupsparse.so")
    return found


def _cuda_lib_dir(nvcc: str) -> str:
    return str(Path(nvcc).resolve().parent.parent / "lib64")


def sources():
    return sorted(CSRC.glob("*.cu"))


def _headers():
    return sorted(CSRC.glob("*.cuh")) + sorted(INCLUDE.glob("*.h"))


def needs_build() -> bool:
    if not LIB.exists():
        return True
    t = LIB.stat().st_mtime
    return any(p.stat().st_mtime > t for p in list(sources()) + _headers() + [Path(__file__)])


def build_library(force: bool = False, verbose: bool = False, extra_flags=None) -> Path:
    if not force and not needs_build():
        return LIB
    nvcc = _nvcc()
    BUILD.mkdir(exist_ok=True)
    common = [nvcc, "-std=c++17", "-O3", "-lineinfo", *ARCH, "-Xcompiler", "-fPIC", f"-I{INCLUDE}",
              "--expt-relaxed-constexpr", *(extra_flags or [])]

    def compile_one(src: Path):
        obj = BUILD / (src.stem + ".o")
        cmd = common + ["-c", str(src), "-o", str(obj)]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src.name}:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    srcs = sources()
    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(srcs), os.cpu_count() or 4))) as ex:
        objs = list(ex.map(compile_one, srcs))
    tmp = LIB.with_suffix(".so.tmp")
    libdir = _cuda_lib_dir(nvcc)
    cmd = [nvcc, "-shared", *ARCH, "-o", str(tmp), *map(str, objs), "-cudart", "shared",
           f"-L{libdir}", "-Xlinker", f"-rpath,{libdir}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose=True))
