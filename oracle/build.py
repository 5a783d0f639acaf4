"""Compile the C oracle into ``oracle/_build/liboracle.so`` (test infrastructure).

gcc, -O2, OpenMP when available, and ``-ffp-contract=off`` so that no compiler
fuses the oracle's multiply-adds: the same source gives the same doubles on
x86-64 and aarch64.
"""
from __future__ import annotations

import os
import subprocess
import sys
from pathlib import Path

HERE = Path(__file__).resolve().parent
SRC = HERE / "wino_oracle.c"
OUT = HERE / "_build" / "liboracle.so"


def build(force: bool = False, verbose: bool = False) -> Path:
    if OUT.exists() and not force and OUT.stat().st_mtime >= SRC.stat().st_mtime:
        return OUT
    OUT.parent.mkdir(parents=True, exist_ok=True)
    tmp = OUT.with_suffix(f".so.tmp{os.getpid()}")
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
            str(SRC), "-o", str(tmp), "-lm"]
    for extra in (["-fopenmp"], []):
        cmd = base[:1] + extra + base[1:]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if verbose:
            print(" ".join(cmd), r.stdout, r.stderr, file=sys.stderr)
        if r.returncode == 0:
            os.replace(tmp, OUT)
            return OUT
    raise RuntimeError(f"oracle build failed:\n{r.stderr}")


if __name__ == "__main__":
    print(build(force=True, verbose=True))
