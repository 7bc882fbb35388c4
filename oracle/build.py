"""Builds the oracle's shared library from ``espace_oracle.c`` with the host C compiler.

The oracle is test infrastructure: building it is part of ``__graft_entry__.build()`` so
that the checker exists on every machine, but no product code loads it.
"""
from __future__ import annotations

import os
import subprocess

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "espace_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")


def library_path() -> str:
    return os.path.join(_OUT_DIR, "liboracle.so")


def build(force: bool = False) -> str:
    out = library_path()
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(_SRC):
        return out
    os.makedirs(_OUT_DIR, exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    cmd = [os.environ.get("CC", "gcc"), "-O2", "-fno-fast-math", "-ffp-contract=off",
           "-fopenmp", "-shared", "-fPIC", "-std=c11", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force=True))
