"""Builds the oracle's shared library (plain C, gcc) in place.

Test infrastructure: compiled by ``__graft_entry__.build()`` and, when stale,
on first use by ``oracle.lib()``.  The output (``liboracle.so``) is
git-ignored.
"""
from __future__ import annotations

import os
import subprocess

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "agnes_oracle.c")
_HDR = os.path.join(_HERE, "agnes_oracle.h")
LIB_PATH = os.path.join(_HERE, "liboracle.so")


def build_oracle(force: bool = False) -> str:
    """Compiles agnes_oracle.c into liboracle.so when missing or stale."""
    newest_src = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if (not force and os.path.exists(LIB_PATH)
            and os.path.getmtime(LIB_PATH) >= newest_src):
        return LIB_PATH
    tmp = LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=gnu11", "-O2", "-fPIC", "-shared", "-Wall", "-Wextra",
           "-o", tmp, _SRC]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build_oracle(force=True))
