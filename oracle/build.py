"""Compile the CPU oracle (test infrastructure) into oracle/libsmat_oracle.so.

The oracle is a plain C++17 single-threaded program built with
-ffp-contract=off and no fast-math, so every float operation it performs is a
single IEEE binary32 (or binary64) operation. Nothing here touches the CUDA
library.
"""

import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "smat_oracle.cpp")
LIB = os.path.join(HERE, "libsmat_oracle.so")


def build(force: bool = False) -> str:
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + ".tmp.%d" % os.getpid()
    cmd = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fno-fast-math",
           "-Wall", "-Wextra", "-shared", "-fPIC", SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
