"""Compile the float64 CPU oracle into ``oracle/liboracle_nystra.so``.

Test infrastructure only (see ``oracle/__init__.py``).  Plain ``gcc -O2``
with OpenMP and without floating-point contraction, so the x86 and Arm hosts
produce the same bits.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "nystra_oracle.c")
LIB = os.path.join(HERE, "liboracle_nystra.so")


def build(force: bool = False) -> str:
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
           "-std=c11", "-o", tmp, SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
