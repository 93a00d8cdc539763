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
LIB_OMP = os.path.join(OUT_DIR, "libalq_oracle_omp.so")

CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
          "-shared", "-fPIC"]


def _stale(lib: str) -> bool:
    if not os.path.exists(lib):
        return True
    lib_t = os.path.getmtime(lib)
    return any(os.path.getmtime(f) > lib_t for f in (SRC, HDR, __file__))


def needs_build() -> bool:
    return _stale(LIB)


def _compile(lib: str, extra) -> None:
    os.makedirs(OUT_DIR, exist_ok=True)
    tmp = lib + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *CFLAGS, *extra, "-o", tmp, SRC, "-lm"], check=True)
    os.replace(tmp, lib)


def build(force: bool = False) -> str:
    """Build the oracle library if it is missing or stale; return its path."""
    if force or _stale(LIB):
        _compile(LIB, [])
    return LIB


def build_threaded(force: bool = False):
    """The same source built with -fopenmp (the all-core CPU baseline): only
    loops with independent iterations run in parallel and every reduction
    keeps its sequential order, so its results are the plain build's bit
    for bit. Returns its path, or None where the compiler has no OpenMP."""
    if force or _stale(LIB_OMP):
        try:
            _compile(LIB_OMP, ["-fopenmp"])
        except (subprocess.CalledProcessError, OSError):
            return None
    return LIB_OMP


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
    print(build_threaded(force="--force" in sys.argv))
