"""Build the oracle's shared library (test infrastructure, not part of the product).

g++ with -O2 and -ffp-contract=off, so that each floating-point operation of the oracle
is one IEEE operation (no fused multiply-add on any host, x86 or Arm).
"""
from __future__ import annotations

import os
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
LIB = HERE / "liboracle.so"
SOURCES = sorted(HERE.glob("*.cpp"))


def _stale() -> bool:
    if not LIB.exists():
        return True
    t = LIB.stat().st_mtime
    return any(p.stat().st_mtime > t for p in SOURCES + [Path(__file__)])


def compile_library(sources, out: Path) -> Path:
    """Compile the given oracle sources into the shared library `out` (same flags as the
    oracle itself; the planted-mistake tests build altered copies with it)."""
    out = Path(out)
    tmp = out.with_suffix(f".so.tmp{os.getpid()}")
    cmd = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-fPIC", "-shared", *map(str, sources), "-o", str(tmp)]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def build_oracle(force: bool = False) -> Path:
    if not force and not _stale():
        return LIB
    return compile_library(SOURCES, LIB)


if __name__ == "__main__":
    print(build_oracle(force=True))
