"""Compile the C oracle into oracle/_build/libalq_oracle.so.

TEST INFRASTRUCTURE (see alq_oracle.h). The flags are part of the oracle's
arithmetic contract: no fast-math, and no multiply-add contraction, so every
fp32 expression rounds after each operation on every host architecture.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "alq_oracle.c")
HDR = os.path.join(HERE, "alq_oracle.h")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libalq_oracle.so")

CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
          "-shared", "-fPIC"]


def needs_build() -> bool:
    if not os.path.exists(LIB):
        return True
    lib_t = os.path.getmtime(LIB)
    return any(os.path.getmtime(f) > lib_t for f in (SRC, HDR, __file__))


def build(force: bool = False) -> str:
    """Build the oracle library if it is missing or stale; return its path."""
    if force or needs_build():
        os.makedirs(OUT_DIR, exist_ok=True)
        tmp = LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", *CFLAGS, "-o", tmp, SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
