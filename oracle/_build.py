"""Builds the oracle's shared library with gcc (test infrastructure only).

IEEE fp32/fp64 with no contraction of a*b+c into a fused multiply-add
(-ffp-contract=off) and no fast-math, so every operation rounds once, in the
order the source writes it, on x86-64 and aarch64 alike.
"""
from __future__ import annotations

import os
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
SRC = HERE / "tula_oracle.c"
OUT = HERE / "_tula_oracle.so"
CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def build_oracle(force: bool = False) -> Path:
    if not force and OUT.exists() and OUT.stat().st_mtime >= SRC.stat().st_mtime:
        return OUT
    tmp = OUT.with_suffix(f".{os.getpid()}.tmp")
    cc = os.environ.get("CC", "gcc")
    # OpenMP only spreads the per-tensor parts of oracle_ags_step_threads over threads; without
    # it the same code runs on one thread.
    for extra in (["-fopenmp"], []):
        cmd = [cc, *CFLAGS, *extra, str(SRC), "-o", str(tmp), "-lm"]
        if subprocess.run(cmd, capture_output=True).returncode == 0:
            break
    else:
        subprocess.run(cmd, check=True)
    os.replace(tmp, OUT)
    return OUT


if __name__ == "__main__":
    print(build_oracle(force=True))
