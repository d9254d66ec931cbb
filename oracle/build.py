"""Build the CPU oracle shared library (test infrastructure only).

gcc, plain C11, no fast-math and no floating-point contraction, so that every fp32
operation in the oracle is rounded exactly once in the order it is written.  OpenMP
splits the outer loops of the large products over host threads (orc_set_threads);
every output element is still computed by one thread in the written order.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "liboracle_nmdlm.so")
SOURCES = [os.path.join(HERE, "nmdlm_oracle.c")]
HEADERS = [os.path.join(HERE, "nmdlm_oracle.h")]


def _stale():
    if not os.path.exists(LIB_PATH):
        return True
    t = os.path.getmtime(LIB_PATH)
    return any(os.path.getmtime(p) > t for p in SOURCES + HEADERS + [__file__])


def build(force=False, verbose=False):
    """Compile the oracle if it is missing or older than its sources; return its path."""
    if not force and not _stale():
        return LIB_PATH
    os.makedirs(BUILD_DIR, exist_ok=True)
    tmp = LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", "-fopenmp", "-Wall", "-Wextra", "-o", tmp] + SOURCES + ["-lm"]
    if verbose:
        print(" ".join(cmd))
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
