"""Build ``libgmgsim.so`` (the C-ABI library) for sm_103a with nvcc, in-tree.

The translation units compile in parallel, then link into one shared library
next to this file.  ``python -m paper_2608_15762_gb300.build``.

A rebuild happens when the library is missing or when the stamp stored beside
it (a SHA-256 over every source and header, the nvcc flags, the nvcc version
and the host machine type) differs from the current one; file times are not
consulted, so a library copied in from elsewhere is never trusted on its
modification time alone.
"""
import hashlib
import os
import platform
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "libgmgsim.so")
SOURCES = ["gmgsim_host.cu", "gmgsim_kernels.cu", "gmgsim_full.cu", "gmgsim_inc.cu", "gmgsim_arb.cu",
           "gmgsim_arbw.cu", "gmgest.cu", "gmground.cu"]
HEADERS = ["gmg_layout.h", "gmg_access.h", "gmg_arb.h", "gmg_arbw.h", "gmg_arb_events.h", "gmgsim_sim.cuh", os.path.join("..", "..", "include", "gmgsim.h"),
           os.path.join("..", "..", "include", "gmgest.h"), os.path.join("..", "..", "include", "gmground.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall"]


def nvcc() -> str:
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


STAMP = OUT + ".stamp"


def _nvcc_version() -> str:
    try:
        return subprocess.run([nvcc(), "--version"], capture_output=True, text=True).stdout
    except OSError:
        return "no nvcc"


def stamp() -> str:
    """SHA-256 over the sources, headers, flags, compiler version and machine."""
    h = hashlib.sha256()
    for name in SOURCES + HEADERS:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read() + b"\0")
    h.update(" ".join(ARCH + FLAGS).encode())
    h.update(_nvcc_version().encode())
    h.update(platform.machine().encode())
    return h.hexdigest()


def _stale(want: str) -> bool:
    if not os.path.exists(OUT) or not os.path.exists(STAMP):
        return True
    with open(STAMP) as f:
        return f.read().strip() != want


def build(force: bool = False, verbose: bool = False) -> str:
    want = stamp()
    if not force and not _stale(want):
        if verbose:
            print("libgmgsim.so up to date (stamp %s)" % want[:12])
        return OUT
    print("building libgmgsim.so (stamp %s)" % want[:12], file=sys.stderr)
    objdir = os.path.join(HERE, "_build")
    os.makedirs(objdir, exist_ok=True)
    procs, objs = [], []
    for s in SOURCES:
        o = os.path.join(objdir, s.replace(".cu", ".o"))
        objs.append(o)
        cmd = [nvcc()] + ARCH + FLAGS + ["-c", os.path.join(CSRC, s), "-o", o]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        procs.append((cmd, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)))
    for cmd, p in procs:
        out, _ = p.communicate()
        if p.returncode != 0 or verbose:
            sys.stdout.write(out.decode(errors="replace"))
        if p.returncode != 0:
            raise RuntimeError("nvcc failed: " + " ".join(cmd))
    tmp = OUT + ".tmp%d" % os.getpid()
    subprocess.check_call([nvcc()] + ARCH + ["-shared", "-o", tmp] + objs)
    os.replace(tmp, OUT)
    with open(STAMP, "w") as f:
        f.write(want + "\n")
    return OUT


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
