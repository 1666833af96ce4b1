"""Compile the oracle (plain C) into oracle/_build/libmpadam_oracle.so.

The oracle is test infrastructure; building it is not using it.  Flags keep
the arithmetic IEEE binary32 with no contraction into fused multiply-adds
beyond the explicit fmaf() calls (GCC contracts by default on AArch64).
"""
from __future__ import annotations

import os
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
SRC = HERE / "mpadam_oracle.c"
HDR = HERE / "mpadam_oracle.h"
OUT_DIR = HERE / "_build"
LIB = OUT_DIR / "libmpadam_oracle.so"

CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
          "-fno-unsafe-math-optimizations", "-Wall", "-Wextra"]


def needs_build() -> bool:
    if not LIB.exists():
        return True
    t = LIB.stat().st_mtime
    return any(p.stat().st_mtime > t for p in (SRC, HDR, Path(__file__)))


def build(force: bool = False) -> Path:
    if not force and not needs_build():
        return LIB
    OUT_DIR.mkdir(exist_ok=True)
    tmp = OUT_DIR / f".libmpadam_oracle.{os.getpid()}.so"
    cmd = [os.environ.get("CC", "gcc"), *CFLAGS, str(SRC), "-o", str(tmp), "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
