"""Compile the CPU oracle into oracle/liboracle.so (test infrastructure).

Plain C, -O2, with floating-point contraction off and no fast-math, so every
fp32/fp64 operation in the source is one IEEE operation.  Portable flags
only: the same source builds on x86-64 and aarch64 hosts.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "asmv_oracle.c")
LIB = os.path.join(HERE, "liboracle.so")


def compile_library(src: str, out: str) -> str:
    """Compile an oracle source file (this one, or an edited copy) to `out`."""
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-Wall", "-Wextra", "-o", out, src, "-lm"]
    subprocess.check_call(cmd)
    return out


def build(force: bool = False) -> str:
    if (not force and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= os.path.getmtime(SRC)):
        return LIB
    tmp = LIB + ".tmp.%d" % os.getpid()
    compile_library(SRC, tmp)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
