"""Build the CPU oracle shared library (test infrastructure only).

Compiles zo_oracle.c with plain IEEE semantics: no contraction of a*b+c into
fused multiply-adds and no fast-math, so every float operation rounds once.
"""
import os
import platform
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "zo_oracle.c")
LIB = os.path.join(HERE, "liboracle.so")
STAMP = LIB + ".arch"


def build(force: bool = False) -> str:
    arch_ok = os.path.exists(STAMP) and open(STAMP).read().strip() == platform.machine()
    if not force and arch_ok and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fno-strict-aliasing",
           "-fPIC", "-shared", "-o", tmp, SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    with open(STAMP, "w") as f:
        f.write(platform.machine())
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
