"""Build the CPU oracle (test infrastructure) as a shared library with g++.

Usage: ``python oracle/build.py``.  Produces ``oracle/liboracle_sim.so`` next
to this file.  Plain C++17, no CUDA, nothing shared with the product library.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "sim_ref.cpp")
OUT = os.path.join(HERE, "liboracle_sim.so")


def build(force: bool = False) -> str:
    if not force and os.path.exists(OUT) and os.path.getmtime(OUT) >= os.path.getmtime(SRC):
        return OUT
    tmp = OUT + ".tmp%d" % os.getpid()
    cmd = ["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-pthread", "-Wall", SRC, "-o", tmp]
    subprocess.check_call(cmd)
    os.replace(tmp, OUT)
    return OUT


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
