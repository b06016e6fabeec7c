"""Builds libgroupsparse.so (the C-ABI library) in-tree with nvcc for sm_103a.

Each translation unit is compiled in parallel to an object under
`paper_2609_33977_gb300/_build/`, then linked into
`paper_2609_33977_gb300/libgroupsparse.so` against the shared CUDA runtime.
Beside the library a stamp file records a hash of every source, header, this
script, the compiler flags and the nvcc version; the library is rebuilt unless
the stamp matches, so a prebuilt library from another tree or another set of
flags is never reused.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
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


STAMP = LIB.with_suffix(".so.stamp")
FLAGS = ["-std=c++17", "-O3", "-lineinfo", *ARCH, "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr"]


def _nvcc_version(nvcc: str) -> str:
    r = subprocess.run([nvcc, "--version"], capture_output=True, text=True)
    return r.stdout.strip()


def build_stamp(extra_flags=None) -> str:
    """Hash of everything the library is built from."""
    h = hashlib.sha256()
    for p in list(sources()) + _headers() + [Path(__file__)]:
        h.update(p.name.encode())
        h.update(p.read_bytes())
    h.update(" ".join(FLAGS + list(extra_flags or [])).encode())
    h.update(_nvcc_version(_nvcc()).encode())
    return h.hexdigest()


def needs_build(extra_flags=None) -> bool:
    if not LIB.exists() or not STAMP.exists():
        return True
    return STAMP.read_text().strip() != build_stamp(extra_flags)


def build_library(force: bool = False, verbose: bool = False, extra_flags=None) -> Path:
    if not force and not needs_build(extra_flags):
        return LIB
    nvcc = _nvcc()
    stamp = build_stamp(extra_flags)
    BUILD.mkdir(exist_ok=True)
    common = [nvcc, *FLAGS, f"-I{INCLUDE}", *(extra_flags or [])]

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
           f"-L{libdir}", "-lcublas", "-Xlinker", f"-rpath,{libdir}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    STAMP.write_text(stamp + "\n")
    return LIB


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose=True))
