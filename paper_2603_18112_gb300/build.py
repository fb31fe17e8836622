"""Builds libtula_ags.so in-tree with nvcc for sm_103a (GB300)."""
from __future__ import annotations

import os
import shutil
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
ROOT = HERE.parent
SRC = HERE / "csrc" / "tula_ags.cu"
HEADER = ROOT / "include" / "tula_ags.h"
LIB = HERE / "libtula_ags.so"

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "-shared",
              "-cudart", "shared", "-fmad=false"]


def cuda_lib_dir(nvcc: str) -> str:
    """The toolkit's library directory (CUDA_HOME/lib64, else next to nvcc's bin/): the shared
    CUDA runtime the library links is found there at run time."""
    home = os.environ.get("CUDA_HOME") or os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return os.path.join(home, "lib64")


def nvcc_path() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"),
                 os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")):
        if cand and os.path.exists(cand):
            return cand
    raise FileNotFoundError("nvcc not found (set NVCC or CUDA_HOME)")


def _stale() -> bool:
    if not LIB.exists():
        return True
    t = LIB.stat().st_mtime
    return any(p.stat().st_mtime > t for p in (SRC, HEADER))


def build(force: bool = False, verbose: bool = False) -> Path:
    """Compile the CUDA library if it is missing or older than its sources."""
    if not force and not _stale():
        return LIB
    tmp = LIB.with_name(f"{LIB.name}.{os.getpid()}.tmp")
    nvcc = nvcc_path()
    cmd = [nvcc, *ARCH, *NVCC_FLAGS, "-Xlinker", f"-rpath={cuda_lib_dir(nvcc)}",
           "-I", str(ROOT / "include"), str(SRC), "-o", str(tmp)]
    if verbose:
        cmd.insert(1, "-Xptxas=-v")
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    import sys
    print(build(force=True, verbose="-v" in sys.argv))
