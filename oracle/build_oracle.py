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
LIB_OMP = os.path.join(HERE, "liboracle_omp.so")  # the same loops, run on all host cores


def build(force=False, verbose=False, parallel=False):
    """Builds liboracle.so (serial), or with parallel=True liboracle_omp.so (-fopenmp, for
    timing the oracle on all host cores only)."""
    lib = LIB_OMP if parallel else LIB
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= os.path.getmtime(SRC):
        return lib
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           *(["-fopenmp"] if parallel else []), SRC, "-o", lib + ".tmp", "-lm"]
    if verbose:
        print(" ".join(cmd), file=sys.stderr)
    subprocess.run(cmd, check=True)
    os.replace(lib + ".tmp", lib)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
    print(build(force="--force" in sys.argv, verbose=True, parallel=True))
