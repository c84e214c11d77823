"""Build the CPU oracle (test infrastructure) as a shared library with g++.

Usage: ``python oracle/build.py``.  Produces ``oracle/liboracle_sim.so`` next
to this file.  Plain C++17, no CUDA, nothing shared with the product library.
"""
import hashlib
import os
import platform
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "sim_ref.cpp")
OUT = os.path.join(HERE, "liboracle_sim.so")


FLAGS = ["-O2", "-std=c++17", "-shared", "-fPIC", "-pthread", "-Wall"]
STAMP = OUT + ".stamp"


def stamp() -> str:
    """SHA-256 over the source, the flags and the machine type: the library is
    rebuilt whenever it differs from the stamp stored beside it."""
    h = hashlib.sha256()
    with open(SRC, "rb") as f:
        h.update(f.read())
    h.update(" ".join(FLAGS).encode() + platform.machine().encode())
    return h.hexdigest()


def build(force: bool = False) -> str:
    want = stamp()
    if not force and os.path.exists(OUT) and os.path.exists(STAMP):
        with open(STAMP) as f:
            if f.read().strip() == want:
                return OUT
    tmp = OUT + ".tmp%d" % os.getpid()
    subprocess.check_call(["g++"] + FLAGS + [SRC, "-o", tmp])
    os.replace(tmp, OUT)
    with open(STAMP, "w") as f:
        f.write(want + "\n")
    return OUT


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
