"""Compile the CPU oracle (bigcn_oracle.c) into oracle/_build/liboracle.so.

Test infrastructure: the library is built with plain -O2, no fast-math and no
floating-point contraction, so that every expression rounds exactly as it is
written in the C source on any host (x86-64 or aarch64).
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "bigcn_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "liboracle.so")

CFLAGS = ["-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
          "-shared", "-Wall", "-Wextra"]


def build(force: bool = False) -> str:
    """Build liboracle.so if missing or older than its sources; return its path."""
    os.makedirs(OUT_DIR, exist_ok=True)
    srcs = [SRC, os.path.join(HERE, "bigcn_oracle.h")]
    if (not force and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= max(os.path.getmtime(s) for s in srcs)):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *CFLAGS, "-o", tmp, SRC, "-lm"], check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
