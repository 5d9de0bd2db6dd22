"""Compile the plain-C oracle (``ppo.c``) into ``oracle/_build/libppo.so``.

Test infrastructure: the library is loaded only by the test suite, the smoke
check and the CPU-baseline leg of the benchmark.  Plain gcc, ``-O2`` (no
fast-math, so every double operation is IEEE round-to-nearest), OpenMP over
tokens.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "ppo.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libppo.so")


def build(force: bool = False, extra_flags=()) -> str:
    """Build the oracle library (if stale) and return its path."""
    return build_variant(LIB, extra_flags=extra_flags, force=force)


def build_variant(out_path: str, extra_flags=(), force: bool = False) -> str:
    """Build ``ppo.c`` with extra compiler flags into ``out_path``."""
    os.makedirs(os.path.dirname(out_path), exist_ok=True)
    if (not force and os.path.exists(out_path)
            and os.path.getmtime(out_path) >= os.path.getmtime(SRC)):
        return out_path
    tmp = out_path + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-D_DEFAULT_SOURCE", "-fPIC", "-shared", "-fopenmp",
           "-Wall", "-Wextra", *extra_flags, SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out_path)
    return out_path


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
