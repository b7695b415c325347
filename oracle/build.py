"""Compile the oracle (plain C, OpenMP) into oracle/libaio_oracle.so.

IEEE semantics are kept: no -ffast-math, and -ffp-contract=off so a*b+c is
never fused (the oracle's rounding is then the same on x86-64 and aarch64).
``mutant`` builds a deliberately wrong variant for the mutation tests.
"""
from __future__ import annotations

import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "aio_oracle.c")


def build(out: str | None = None, mutant: int = 0, force: bool = False) -> str:
    out = out or os.path.join(HERE, "libaio_oracle.so")
    if not force and mutant == 0 and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(SRC):
        return out
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-ffp-contract=off",
           f"-DAIO_ORACLE_MUTANT={int(mutant)}", SRC, "-o", out, "-lm"]
    subprocess.run(cmd, check=True)
    return out


if __name__ == "__main__":
    print(build(force=True))
