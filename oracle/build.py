"""Compiles the oracle (test infrastructure) into oracle/libmlkv_oracle.so with the host C compiler.

No FMA contraction (-ffp-contract=off), so the oracle's rounding is the same on x86_64 and aarch64.
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "mlkv_oracle.c")
LIB = os.path.join(HERE, "libmlkv_oracle.so")


def command():
    cc = os.environ.get("CC", "gcc")
    return [cc, "-std=c99", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
            "-D_POSIX_C_SOURCE=200809L", "-o", LIB, SRC, "-lm", "-lpthread"]


def needs_build():
    return (not os.path.exists(LIB)) or os.path.getmtime(LIB) < os.path.getmtime(SRC)


def build(force=False):
    if force or needs_build():
        subprocess.run(command(), check=True)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
