"""Compile the reference oracle (test infrastructure) into a shared library.

The oracle is plain C11 built with gcc; -ffp-contract=off keeps every
binary64 operation separately rounded, so results are the same on x86-64
and aarch64 hosts.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "lc_oracle.c")
LIB = os.path.join(HERE, "liblc_oracle.so")


def build_oracle(force: bool = False) -> str:
    """Build oracle/liblc_oracle.so if missing or older than its source."""
    hdr = os.path.join(HERE, "lc_oracle.h")
    if (not force and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= max(os.path.getmtime(SRC), os.path.getmtime(hdr))):
        return LIB
    tmp = LIB + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-Wall", "-Wextra", "-o", tmp, SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build_oracle(force="--force" in sys.argv))
