"""Compiles the C part of the oracle (layer_math.c) into oracle/liboracle.so.

The oracle is test infrastructure; building it is not using it. Plain gcc, no flags that
change floating-point semantics (-ffp-contract=off keeps every multiply and add rounded
on its own, on x86_64 and aarch64 alike)."""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "layer_math.c")
LIB = os.path.join(HERE, "liboracle.so")


def build(force=False, verbose=False):
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           SRC, "-o", LIB + ".tmp", "-lm"]
    if verbose:
        print(" ".join(cmd), file=sys.stderr)
    subprocess.run(cmd, check=True)
    os.replace(LIB + ".tmp", LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
