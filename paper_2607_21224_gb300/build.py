"""Build libcpdp.so in-tree with nvcc for GB300 (sm_103a).

The library is plain CUDA C++ with a C ABI (include/cpdp.h); it links the
CUDA runtime statically, so loading it needs only the NVIDIA driver.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from pathlib import Path

PKG = Path(__file__).resolve().parent
ROOT = PKG.parent
INCLUDE = ROOT / "include"
CSRC = PKG / "csrc"
SOURCES = [CSRC / "cpdp.cu"]
DEPENDS = SOURCES + [CSRC / "cpdp_kernels.cuh", CSRC / "cpdp_shapes.cuh", CSRC / "cpdp_tma.cuh",
                     CSRC / "cpdp_floor.cuh", CSRC / "cpdp_shuffle.cuh", INCLUDE / "cpdp.h"]
LIBRARY = PKG / "libcpdp.so"
CHECKED_LIBRARY = PKG / "libcpdp_checked.so"  # debug build: kernels count out-of-range indices
BUILD_DIR = ROOT / "_build"
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc_path() -> str:
    found = shutil.which("nvcc")
    if found:
        return found
    cand = Path(os.environ.get("CUDA_HOME", "/usr/local/cuda")) / "bin" / "nvcc"
    if cand.exists():
        return str(cand)
    raise RuntimeError("nvcc not found (set CUDA_HOME or put nvcc on PATH)")


def nvcc_command(output: Path, sources=SOURCES, extra: list[str] | None = None) -> list[str]:
    return [nvcc_path(), "-O3", "-std=c++17", *ARCH, "-lineinfo",
            "-Xcompiler", "-fPIC,-O2", "-shared", "-Xptxas", "-v",
            f"-I{INCLUDE}", f"-I{CSRC}", "-o", str(output), *map(str, sources), *(extra or [])]


def is_stale(output: Path = LIBRARY) -> bool:
    if not output.exists():
        return True
    built = output.stat().st_mtime
    return any(dep.stat().st_mtime > built for dep in DEPENDS)


def build_library(force: bool = False, verbose: bool = False, checked: bool = False) -> Path:
    """Compile libcpdp.so if it is missing or older than its sources. The ptxas
    report (registers, spills, shared memory per kernel) goes to _build/ptxas.txt.
    With `checked`, the debug build libcpdp_checked.so instead (-DCPDP_CHECKED:
    every kernel index is checked against its buffer's extent; report in
    _build/ptxas_checked.txt)."""
    out = CHECKED_LIBRARY if checked else LIBRARY
    if not force and not is_stale(out):
        return out
    BUILD_DIR.mkdir(exist_ok=True)
    tmp = out.with_name(f".{out.stem}.{os.getpid()}.so")
    proc = subprocess.run(nvcc_command(tmp, extra=["-DCPDP_CHECKED"] if checked else None),
                          capture_output=True, text=True)
    (BUILD_DIR / ("ptxas_checked.txt" if checked else "ptxas.txt")).write_text(proc.stdout + proc.stderr)
    if proc.returncode != 0:
        raise RuntimeError(f"nvcc failed ({proc.returncode}):\n{proc.stderr[-4000:]}")
    if verbose:
        print(proc.stderr)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build_library(force=True, verbose=True))
