"""Build the CPU oracle (test infrastructure) with gcc.

Produces ``oracle/_build/liboracle.so`` from ``dpo_oracle.c``: plain C11,
-O2 without fast-math (IEEE double arithmetic, default rounding), OpenMP over
the element loops. Run ``python oracle/build.py`` or call :func:`build`.
"""
from __future__ import annotations

import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "dpo_oracle.c")
HDR = os.path.join(HERE, "dpo_oracle.h")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "liboracle.so")


def _stale(lib: str, sources) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    return any(os.path.getmtime(s) > t for s in sources)


def build(force: bool = False, src: str = SRC, out: str = LIB) -> str:
    """Compile the oracle if it is missing or older than its sources."""
    if not force and not _stale(out, [src, HDR]):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-ffp-contract=off", "-Wall", "-Wextra",
           "-I", HERE, src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
