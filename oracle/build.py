"""Compile the fp64 CPU oracle (test infrastructure) into oracle/liboracle_cola.so.

Plain gcc, OpenMP, no fast-math and no FMA contraction, so each sum is the
sequential fp64 sum the oracle's source spells out, on x86 and Arm alike.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "cola_oracle.c")
LIB = os.path.join(HERE, "liboracle_cola.so")


def build(force: bool = False) -> str:
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    cmd = ["gcc", "-O2", "-std=c11", "-D_GNU_SOURCE", "-ffp-contract=off", "-fopenmp",
           "-fPIC", "-shared", "-o", LIB + ".tmp", SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(LIB + ".tmp", LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
