"""Build ``libadpsgd.so`` (the C ABI of include/adpsgd.h) in-tree for sm_103a.

Every .cu file in csrc/ is compiled by nvcc for sm_103a only, with IEEE division and square
root, no flush-to-zero and no multiply-add contraction (the generator and the update are
specified operation by operation); every .cpp file is host C++.  The objects are compiled in
parallel and linked by nvcc with the static CUDA runtime.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libadpsgd.so")
INCLUDE = os.path.join(ROOT, "include")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-fmad=false", "-prec-div=true",
              "-prec-sqrt=true", "-ftz=false", "-Xcompiler", "-ffp-contract=off", "-Xptxas", "-v"]
CXX_FLAGS = ["-O2", "-std=c++17", "-fPIC", "-ffp-contract=off", "-fno-fast-math", "-Wall", "-Wextra"]


def _cuda_home() -> str:
    for cand in (os.environ.get("CUDA_HOME"), "/usr/local/cuda"):
        if cand and os.path.exists(os.path.join(cand, "bin", "nvcc")):
            return cand
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(nvcc))
    raise RuntimeError("nvcc not found: the CUDA library cannot be built")


def _sources():
    return [os.path.join(CSRC, f) for f in sorted(os.listdir(CSRC))] + [os.path.join(INCLUDE, "adpsgd.h")]


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in _sources())


def _run(cmd, log):
    r = subprocess.run(cmd, capture_output=True, text=True)
    with open(log, "w") as f:
        f.write(" ".join(cmd) + "\n" + r.stdout + r.stderr)
    if r.returncode != 0:
        sys.stderr.write(r.stdout + r.stderr)
        raise RuntimeError(f"build step failed: {' '.join(cmd)}")


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile and link the library if any source is newer than it; return its path."""
    if not force and not _stale():
        return LIB
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    os.makedirs(BUILD, exist_ok=True)
    jobs, objs = [], []
    for f in sorted(os.listdir(CSRC)):
        src = os.path.join(CSRC, f)
        stem, ext = os.path.splitext(f)
        obj = os.path.join(BUILD, stem + ".o")
        if ext == ".cu":
            jobs.append(([nvcc, *ARCH, *NVCC_FLAGS, "-I", INCLUDE, "-c", src, "-o", obj],
                         os.path.join(BUILD, stem + ".log")))
        elif ext == ".cpp":
            jobs.append((["g++", *CXX_FLAGS, "-I", os.path.join(cuda, "include"), "-I", INCLUDE, "-c", src, "-o", obj],
                         os.path.join(BUILD, stem + ".log")))
        else:
            continue
        objs.append(obj)
    with ThreadPoolExecutor(len(jobs)) as ex:
        for fut in [ex.submit(_run, c, l) for c, l in jobs]:
            fut.result()
    tmp = LIB + f".tmp{os.getpid()}"
    _run([nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"], os.path.join(BUILD, "link.log"))
    os.replace(tmp, LIB)
    if verbose:
        for f in sorted(os.listdir(BUILD)):
            if f.endswith(".log") and f != "link.log":
                with open(os.path.join(BUILD, f)) as fh:
                    sys.stdout.write(fh.read())
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
