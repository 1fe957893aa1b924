"""Compile the fp64 CPU oracle (test infrastructure) into oracle/_build/liboracle.so.

Plain C, -O2, no fast-math, OpenMP for splitting independent output rows. Builds the same
way on x86_64 and aarch64 (no architecture flags).
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "resbm_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "liboracle.so")


def build(force: bool = False, src: str = SRC, out: str = LIB) -> str:
    """Compile the oracle unless an up-to-date library exists; return its path.

    `src`/`out` let a test compile a modified copy (a planted mistake) somewhere else.
    """
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if (not force and src == SRC and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(SRC)):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
           src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
