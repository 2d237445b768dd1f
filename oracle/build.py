"""Builds the oracle's shared library (plain C, gcc, OpenMP) in-tree.

Test infrastructure only: the CUDA library's build never touches this file.
"""
from __future__ import annotations

import os
import subprocess
import sys

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lla_oracle.c")


def library_path() -> str:
    return os.path.join(_HERE, "liblla_oracle.so")


def build_oracle(force: bool = False) -> str:
    """Compiles lla_oracle.c into liblla_oracle.so unless an up-to-date copy exists."""
    out = library_path()
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(_SRC)):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-Wall", "-Wextra",
           _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build_oracle(force="--force" in sys.argv))
